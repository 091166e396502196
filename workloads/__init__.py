"""Seeded synthetic workloads shared by the tests, the bench and the oracle checks.

This module only describes shapes and draws random inputs; it holds none of the
method's arithmetic (no quantisation, no dequantisation, no matmul), so that the
CUDA path and the CPU oracle can both be fed from it without sharing code.

The paper evaluates closed-loop policies whose weights and tasks are not
available here (Section 4, Tables 3-4), so every input is synthetic: weights
~N(0, 0.02) in fp32 (optionally with 1% of entries multiplied by 8), activations
~N(0, 1) rounded to bf16.  The token counts follow one closed-loop step of the
paper's batch-1 closed-loop setting (Section 3.1, challenge 2):
M=1 action-token decode, M=50 action-chunk denoising, M=280..816 prefix prefill.
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional, Sequence

import numpy as np

Q8_0 = 0
Q4_0 = 1
Q6_0 = 2
FMT_NAMES = {Q8_0: "Q8_0", Q4_0: "Q4_0", Q6_0: "Q6_0"}
BLOCK_BYTES = {Q8_0: 34, Q4_0: 18, Q6_0: 26}   # packed bytes per 32 weights (codes + fp16 scale)


# layer epilogues (the library's emb_epilogue values)
EPI_F32, EPI_BF16, EPI_ADD, EPI_GEGLU, EPI_SWIGLU = 0, 1, 2, 3, 4


def output_bytes(epilogue: int, M: int, N: int) -> int:
    """Bytes a layer's output moves: fp32 write, bf16 write, fp32 read + write (residual
    add), or one bf16 per gate/up row pair."""
    return {EPI_F32: 4 * M * N, EPI_BF16: 2 * M * N, EPI_ADD: 8 * M * N,
            EPI_GEGLU: M * N, EPI_SWIGLU: M * N}[epilogue]


@dataclasses.dataclass(frozen=True)
class Linear:
    """One weight matrix W [N][K] (PyTorch Linear.weight layout)."""
    name: str
    N: int
    K: int
    seed: int
    outliers: float = 0.0  # fraction of weights multiplied by 8 before quantisation
    epilogue: int = EPI_F32
    # the layer's X is the output of the group this many groups earlier (0: its own input)
    x_from: int = 0


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    fmt: int
    M: int
    layers: int
    # linears of one layer, grouped by stage: the linears inside a group read the same
    # activation (q/k/v, gate/up); a group only starts once the previous group is done.
    groups: Sequence[Sequence[Linear]]
    repeats: int = 1  # passes over the same weights (denoising steps)

    def linears(self) -> List[Linear]:
        return [lin for g in self.groups for lin in g]

    @property
    def params(self) -> int:
        return sum(l.N * l.K for l in self.linears())

    def weight_bytes(self) -> int:
        per = BLOCK_BYTES[self.fmt]
        return sum(l.N * l.K // 32 * per for l in self.linears())

    def algorithmic_bytes(self) -> int:
        """Weights read once + X read once (bf16) + the output per the layer's epilogue
        (fp32 written once unless fused), per pass."""
        return self.weight_bytes() + sum(self.M * l.K * 2 + output_bytes(l.epilogue, self.M, l.N)
                                         for l in self.linears())

    def flops(self) -> int:
        return sum(2 * self.M * l.N * l.K for l in self.linears())


def _decoder_layers(prefix: str, n_layers: int, hidden: int, kv: int, ffn: int,
                    seed_base: int, outliers: float = 0.0, q: Optional[int] = None):
    q = hidden if q is None else q
    groups = []
    for layer in range(n_layers):
        s = seed_base + 16 * layer
        groups.append([Linear(f"{prefix}{layer}.q", q, hidden, s + 0, outliers),
                       Linear(f"{prefix}{layer}.k", kv, hidden, s + 1, outliers),
                       Linear(f"{prefix}{layer}.v", kv, hidden, s + 2, outliers)])
        groups.append([Linear(f"{prefix}{layer}.o", hidden, q, s + 3, outliers)])
        groups.append([Linear(f"{prefix}{layer}.gate", ffn, hidden, s + 4, outliers),
                       Linear(f"{prefix}{layer}.up", ffn, hidden, s + 5, outliers)])
        groups.append([Linear(f"{prefix}{layer}.down", hidden, ffn, s + 6, outliers)])
    return groups


def _vit_layers(n_layers: int, width: int, mlp: int, seed_base: int):
    groups = []
    for layer in range(n_layers):
        s = seed_base + 16 * layer
        groups.append([Linear(f"vit{layer}.qkv", 3 * width, width, s + 0)])
        groups.append([Linear(f"vit{layer}.o", width, width, s + 1)])
        groups.append([Linear(f"vit{layer}.fc1", mlp, width, s + 2)])
        groups.append([Linear(f"vit{layer}.fc2", width, mlp, s + 3)])
    return groups


def single_linear() -> Workload:
    """One 2048x2048 Q8_0 linear at M=1."""
    return Workload("single_q8_0_2048x2048_m1", Q8_0, 1, 1,
                    [[Linear("w", 2048, 2048, 1)]])


def single_linear_copies(copies: int = 100) -> Workload:
    """The single 2048x2048 Q8_0 linear at M=1 as a chain of `copies` calls, each on its own
    copy of the weights and activation (seeds 1 .. copies), so that together the copies
    (100 x 4.46 MB) exceed three times the 126 MB L2 and HBM serves every call."""
    return Workload(f"single_q8_0_2048x2048_m1_x{copies}", Q8_0, 1, 1,
                    tuple((Linear(f"w{i}", 2048, 2048, 1 + i),) for i in range(copies)))


def gemma2b_decode(fmt: int) -> Workload:
    """Gemma-style 2B decoder linears, 18 layers, hidden 2048, kv 256, ffn 16384, M=1."""
    return Workload(f"gemma2b_decode_{FMT_NAMES[fmt].lower()}_m1", fmt, 1, 18,
                    _flatten_layers(_decoder_layers("L", 18, 2048, 256, 16384, 1000)))


def action_expert_denoise() -> Workload:
    """Flow-matching action expert: 18 layers, width 1024, M=50, 10 denoising steps."""
    return Workload("action_expert_q8_0_m50_x10", Q8_0, 50, 18,
                    _flatten_layers(_decoder_layers("A", 18, 1024, 128, 4096, 3000)),
                    repeats=10)


def action_expert_fused(steps: int = 10) -> Workload:
    """The action expert's flow-matching loop as one chain: `steps` denoising steps x 18
    layers, M = 50, Q8_0, with fused epilogues: q/k/v write bf16 (the attention's inputs),
    o and down add into one fp32 residual stream, gate/up is one matrix of interleaved
    rows whose GeGLU output (bf16) is down's input."""
    groups = []
    for step in range(steps):
        for layer in range(18):
            s = 3000 + 16 * layer      # the same weights every step
            a = f"A{layer}"
            groups.append([Linear(f"{a}.q", 1024, 1024, s + 0, epilogue=EPI_BF16),
                           Linear(f"{a}.k", 128, 1024, s + 1, epilogue=EPI_BF16),
                           Linear(f"{a}.v", 128, 1024, s + 2, epilogue=EPI_BF16)])
            groups.append([Linear(f"{a}.o", 1024, 1024, s + 3, epilogue=EPI_ADD)])
            groups.append([Linear(f"{a}.gate_up", 2 * 4096, 1024, s + 4, epilogue=EPI_GEGLU)])
            groups.append([Linear(f"{a}.down", 1024, 4096, s + 6, epilogue=EPI_ADD, x_from=1)])
    return Workload(f"action_expert_fused_q8_0_m50_x{steps}", Q8_0, 50, 18 * steps,
                    _flatten_layers(groups))


def gemma2b_prefill(fmt: int) -> Workload:
    """Backbone prefill over 3x256 image + 48 text tokens (M=816)."""
    return Workload(f"gemma2b_prefill_{FMT_NAMES[fmt].lower()}_m816", fmt, 816, 18,
                    _flatten_layers(_decoder_layers("L", 18, 2048, 256, 16384, 1000)))


def vit_tower(fmt: int) -> Workload:
    """ViT-style vision tower, width 1152, 27 layers, M=768."""
    return Workload(f"vit_{FMT_NAMES[fmt].lower()}_m768", fmt, 768, 27,
                    _flatten_layers(_vit_layers(27, 1152, 4608, 5000)))


def llama7b(M: int) -> Workload:
    """Llama-style 7B backbone, 32 layers, hidden 4096, ffn 11008, Q4_0 with 1% outliers."""
    return Workload(f"llama7b_q4_0_m{M}", Q4_0, M, 32,
                    _flatten_layers(_decoder_layers("L", 32, 4096, 4096, 11008, 7000,
                                                    outliers=0.01)))


def _flatten_layers(groups):
    return tuple(tuple(g) for g in groups)


def all_workloads() -> List[Workload]:
    return [single_linear(), gemma2b_decode(Q8_0), gemma2b_decode(Q4_0),
            action_expert_denoise(), gemma2b_prefill(Q8_0), gemma2b_prefill(Q4_0),
            vit_tower(Q8_0), vit_tower(Q4_0), llama7b(1), llama7b(280)]


# --------------------------------------------------------------------------- generators

def weight_torch(lin: Linear, device="cpu"):
    """fp32 W [N][K] ~ N(0, 0.02) from lin.seed (torch generator on `device`)."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(lin.seed)
    w = torch.randn(lin.N, lin.K, generator=g, device=device, dtype=torch.float32) * 0.02
    if lin.outliers > 0:
        mask = torch.rand(lin.N, lin.K, generator=g, device=device) < lin.outliers
        w = torch.where(mask, w * 8.0, w)
    return w


def activation_torch(M: int, K: int, seed: int, device="cpu"):
    """bf16 X [M][K]: ~N(0, 1) drawn in fp32 and rounded to bf16 (round to nearest even)."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return torch.randn(M, K, generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)


def activation_seed(lin: Linear, step: int = 0) -> int:
    return 1_000_003 * (step + 1) + lin.seed


def weight_np(N: int, K: int, seed: int, scale: float = 0.02) -> np.ndarray:
    return (np.random.default_rng(seed).standard_normal((N, K)) * scale).astype(np.float32)


def bf16_bits_np(x: np.ndarray) -> np.ndarray:
    """bf16 bit patterns of fp32 values via torch's conversion (input preparation only)."""
    import torch
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def activation_bits_np(M: int, K: int, seed: int) -> np.ndarray:
    x = np.random.default_rng(seed).standard_normal((M, K)).astype(np.float32)
    return bf16_bits_np(x)


@dataclasses.dataclass(frozen=True)
class LayerLoop:
    """Whole transformer layers run as a loop (the action expert's flow-matching steps):
    per step, `layers` layers of RMSNorm -> q/k/v (bf16) -> rotary -> attention over the
    layer's prefix key/value cache plus the chunk's own keys -> o (+ residual) -> RMSNorm ->
    gate/up (interleaved rows, GeGLU, bf16) -> down (+ residual). Every step reuses the
    layers' weights, caches and buffers."""
    name: str
    fmt: int
    M: int          # chunk tokens
    D: int          # width
    H: int          # query heads
    Hk: int         # key/value heads
    d: int          # head dim
    F: int          # ffn width (gate/up has 2F interleaved rows)
    prefix: int     # prefix cache tokens (the chunk sits at positions prefix .. prefix + M - 1)
    layers: int
    steps: int
    seed0: int

    def linears(self, layer: int):
        """The layer's matrices: q, k, v, o, gate_up (2F interleaved rows), down."""
        s = self.seed0 + 16 * layer
        a = f"{self.name}.L{layer}"
        return [Linear(f"{a}.q", self.H * self.d, self.D, s + 0),
                Linear(f"{a}.k", self.Hk * self.d, self.D, s + 1),
                Linear(f"{a}.v", self.Hk * self.d, self.D, s + 2),
                Linear(f"{a}.o", self.D, self.H * self.d, s + 3),
                Linear(f"{a}.gate_up", 2 * self.F, self.D, s + 4),
                Linear(f"{a}.down", self.D, self.F, s + 6)]

    def layer_flops(self) -> int:
        mm = sum(2 * self.M * lin.N * lin.K for lin in self.linears(0))
        attn = 4 * self.M * self.H * (self.prefix + self.M) * self.d   # q.k and p.v
        return mm + attn

    def layer_bytes(self) -> int:
        """Algorithmic bytes of one layer: weights once, every activation read and written
        once, the prefix cache and the chunk's keys/values read once."""
        M, D, F = self.M, self.D, self.F
        qd, kd = self.H * self.d, self.Hk * self.d
        w = sum(lin.N * lin.K // 32 * BLOCK_BYTES[self.fmt] for lin in self.linears(0))
        norm = 2 * (4 * M * D + 4 * D + 2 * M * D)               # two norms: residual, gamma, out
        qkv = 2 * M * D + 2 * M * (qd + 2 * kd)                  # read h, write q, k, v
        rope = 2 * 2 * M * (qd + kd)                             # q, k read and written
        attn = 2 * M * qd + 2 * 2 * (self.prefix + M) * kd + 2 * M * qd
        o = 2 * M * qd + 8 * M * D                                # read a, residual add
        gu = 2 * M * D + 2 * M * F                                # read h2, write GeGLU output
        down = 2 * M * F + 8 * M * D
        return w + norm + qkv + rope + attn + o + gu + down

    def flops(self) -> int:
        return self.layer_flops() * self.layers * self.steps

    def algorithmic_bytes(self) -> int:
        return self.layer_bytes() * self.layers * self.steps

    def launches(self) -> int:
        """Kernel launches of one loop: norm, q/k/v, rotary of q and k, attention, o, norm,
        gate/up, down per layer."""
        return 8 * self.layers * self.steps


def action_expert_layers(steps: int = 10) -> LayerLoop:
    """The action expert (width 1024, 8 query heads and 1 key/value head of 128, ffn 4096,
    18 layers) over an 816-token prefix cache (3 x 256 image + 48 text tokens), M = 50,
    Q8_0, 10 denoising steps."""
    return LayerLoop("action_expert_layers", Q8_0, 50, 1024, 8, 1, 128, 4096, 816, 18, steps, 7000)
