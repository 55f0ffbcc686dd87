"""Seeded synthetic GEMM sets (inputs only; no GEMM arithmetic in here).

This module is the one place both the product path and the CPU oracle get
their inputs from: it draws bf16 matrices from a seeded ``torch.Generator``
on the CPU and hands them out as tensors and as raw uint16 bit patterns, so
both sides read identical bits.  It imports nothing else from the package.

The sets stand in for the paper's GEMMs from low-batch RNNs, Transformers and
tensor-sliced layers (Sec. 5.2, Table "apps"); the paper's own list of 410 /
1072 GEMM sizes is not available, so these shapes follow the workload
families it describes:

* ``pair_256``    — 2 x (M=256, N=256, K=512), U[-1, 1], seed 0, fp32 out.
* ``ffn_slices``  — tensor-sliced Transformer FFN at low batch:
                    4 x (M=128 tokens, N=1024, K=4096), N(0, 0.02), seed 1,
                    bf16 out.
* ``lstm_gates``  — LSTM gate GEMMs at small batch: 8 x (M=32, N=4096,
                    K=1024), U[-0.1, 0.1], seed 2, fp32 out.
* ``hetero_pair`` — two co-running models: 3 x (512, 1024, 1024) plus
                    1 x (2048, 8192, 2048), N(0, 1/sqrt(K)), seed 3, fp32 out.
* ``sweep``       — 64 sets of 2-16 GEMMs, M log-uniform in [16, 4096],
                    N and K log-uniform in [256, 8192] rounded to multiples of
                    64, U[-1, 1], fp32 out; set j uses seed 1000 + j.
* batched study   — sets of 2 or 4 strided-batched attention GEMMs over
                    variable sequence lengths (``make_batched_set``).

Drawing order (fixed, so a set is reproducible from its seed): for GEMM i in
order, A_i (M x K) then B_i (K x N), each as fp32 values rounded to bf16
(round to nearest even).  ``uniform[a, b]`` is ``a + (b - a) * rand``;
``normal(0, s)`` is ``s * randn``.  For the sweep, the set's size and all
shapes are drawn first from the same generator, then the values.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import List, Optional, Tuple

import numpy as np
import torch

DTYPE_BF16 = 0
DTYPE_F32 = 1


@dataclass(frozen=True)
class GemmSpec:
    M: int
    N: int
    K: int
    out_dtype: int              # DTYPE_BF16 or DTYPE_F32
    dist: str                   # "uniform" or "normal"
    scale: float                # half-width for uniform, std-dev for normal
    batch: int = 1              # strided batch entries (A: batch x M x K, B: batch x K x N)

    @property
    def flops(self) -> int:
        return 2 * self.M * self.N * self.K * self.batch

    @property
    def bytes(self) -> int:
        """Algorithmic bytes: A and B read once, C written once."""
        out = 2 if self.out_dtype == DTYPE_BF16 else 4
        return self.batch * (2 * self.M * self.K + 2 * self.K * self.N + out * self.M * self.N)


@dataclass
class GemmSet:
    name: str
    seed: int
    specs: List[GemmSpec]
    a: List[torch.Tensor] = field(default_factory=list)   # bf16, CPU, M x K
    b: List[torch.Tensor] = field(default_factory=list)   # bf16, CPU, K x N

    @property
    def flops(self) -> int:
        return sum(s.flops for s in self.specs)

    @property
    def bytes(self) -> int:
        return sum(s.bytes for s in self.specs)

    def a_bits(self, i: int) -> np.ndarray:
        return bits_of(self.a[i])

    def b_bits(self, i: int) -> np.ndarray:
        return bits_of(self.b[i])


def bits_of(t: torch.Tensor) -> np.ndarray:
    """Raw uint16 bit patterns of a bf16 CPU tensor (no copy of values)."""
    assert t.dtype == torch.bfloat16
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


def _draw(gen: torch.Generator, rows: int, cols: int, dist: str, scale: float) -> torch.Tensor:
    if dist == "uniform":
        x = torch.rand((rows, cols), generator=gen, dtype=torch.float32)
        x = -scale + (2.0 * scale) * x
    elif dist == "normal":
        x = scale * torch.randn((rows, cols), generator=gen, dtype=torch.float32)
    else:
        raise ValueError(dist)
    return x.to(torch.bfloat16)


def materialize(name: str, seed: int, specs: List[GemmSpec],
                gen: Optional[torch.Generator] = None) -> GemmSet:
    if gen is None:
        gen = torch.Generator(device="cpu")
        gen.manual_seed(seed)
    s = GemmSet(name, seed, list(specs))
    for sp in specs:
        if sp.batch == 1:
            s.a.append(_draw(gen, sp.M, sp.K, sp.dist, sp.scale))
            s.b.append(_draw(gen, sp.K, sp.N, sp.dist, sp.scale))
        else:   # entry by entry: A_i then B_i
            a, b = [], []
            for _ in range(sp.batch):
                a.append(_draw(gen, sp.M, sp.K, sp.dist, sp.scale))
                b.append(_draw(gen, sp.K, sp.N, sp.dist, sp.scale))
            s.a.append(torch.stack(a))
            s.b.append(torch.stack(b))
    return s


def config_specs(name: str) -> Tuple[int, List[GemmSpec]]:
    """(seed, GEMM specs) of a named fixed configuration."""
    if name == "pair_256":
        return 0, [GemmSpec(256, 256, 512, DTYPE_F32, "uniform", 1.0)] * 2
    if name == "ffn_slices":
        return 1, [GemmSpec(128, 1024, 4096, DTYPE_BF16, "normal", 0.02)] * 4
    if name == "lstm_gates":
        return 2, [GemmSpec(32, 4096, 1024, DTYPE_F32, "uniform", 0.1)] * 8
    if name == "hetero_pair":
        small = GemmSpec(512, 1024, 1024, DTYPE_F32, "normal", 1.0 / math.sqrt(1024))
        big = GemmSpec(2048, 8192, 2048, DTYPE_F32, "normal", 1.0 / math.sqrt(2048))
        return 3, [small, small, small, big]
    raise KeyError(name)


FIXED_CONFIGS = ("pair_256", "ffn_slices", "lstm_gates", "hetero_pair")
SWEEP_SETS = 64


def make_config(name: str) -> GemmSet:
    seed, specs = config_specs(name)
    return materialize(name, seed, specs)


def _log_uniform(gen: torch.Generator, lo: float, hi: float) -> float:
    u = float(torch.rand((1,), generator=gen, dtype=torch.float64)[0])
    return math.exp(math.log(lo) + u * (math.log(hi) - math.log(lo)))


def sweep_specs(j: int) -> Tuple[int, List[GemmSpec], torch.Generator]:
    """Shapes of sweep set j (0 <= j < 64) and the generator positioned for
    drawing its values."""
    seed = 1000 + j
    gen = torch.Generator(device="cpu")
    gen.manual_seed(seed)
    n = 2 + int(torch.randint(0, 15, (1,), generator=gen)[0])      # 2..16
    specs = []
    for _ in range(n):
        M = int(round(_log_uniform(gen, 16, 4096)))
        M = min(max(M, 16), 4096)
        N = 64 * int(round(_log_uniform(gen, 256, 8192) / 64))
        N = min(max(N, 256), 8192)
        K = 64 * int(round(_log_uniform(gen, 256, 8192) / 64))
        K = min(max(K, 256), 8192)
        specs.append(GemmSpec(M, N, K, DTYPE_F32, "uniform", 1.0))
    return seed, specs, gen


def predictor_dataset_shapes(total: int = 1072, seed: int = 5000) -> List[Tuple[int, int, int, int]]:
    """Distinct GEMM shapes (M, N, K, out dtype) for the CD predictor's
    training set: those of the fixed sets and of the 64 randomized sets first,
    then seeded log-uniform draws over the same ranges (M in [16, 4096]; N, K
    multiples of 64 in [256, 8192]; bf16 or fp32 out) up to `total`."""
    out: List[Tuple[int, int, int, int]] = []
    seen = set()

    def add(t):
        if t not in seen and len(out) < total:
            seen.add(t)
            out.append(t)

    for name in FIXED_CONFIGS:
        for s in config_specs(name)[1]:
            add((s.M, s.N, s.K, s.out_dtype))
    for j in range(SWEEP_SETS):
        for s in sweep_specs(j)[1]:
            add((s.M, s.N, s.K, s.out_dtype))
    gen = torch.Generator(device="cpu")
    gen.manual_seed(seed)
    while len(out) < total:
        M = min(max(int(round(_log_uniform(gen, 16, 4096))), 16), 4096)
        N = min(max(64 * int(round(_log_uniform(gen, 256, 8192) / 64)), 256), 8192)
        K = min(max(64 * int(round(_log_uniform(gen, 256, 8192) / 64)), 256), 8192)
        o = int(torch.randint(0, 2, (1,), generator=gen)[0])
        add((M, N, K, DTYPE_BF16 if o == 0 else DTYPE_F32))
    return out


def scaling_study_shapes(stride: int = 16) -> List[Tuple[int, int, int, int]]:
    """GEMM shapes of the GPU-scaling study (every `stride`-th shape of the
    predictor's training set; each runs as a set of 4 equal GEMMs, CD 4)."""
    return predictor_dataset_shapes()[::stride]


def make_scaling_set(i: int, copies: int = 4) -> GemmSet:
    """Set i of the GPU-scaling study: `copies` equal GEMMs, U[-1, 1] inputs,
    seed 3000 + i."""
    M, N, K, out = scaling_study_shapes()[i]
    specs = [GemmSpec(M, N, K, out, "uniform", 1.0) for _ in range(copies)]
    return materialize(f"scaling_{i:02d}", 3000 + i, specs)


def batched_study_specs(i: int, members: int) -> Tuple[int, List[GemmSpec]]:
    """Set i of the batched study: `members` (2 or 4) heterogeneous strided
    batched GEMMs of attention over variable-length inputs (Sec. 6.7's
    B-GEMMs): per member a sequence length L from {128, ..., 2048} and 16 or
    32 heads of dimension 128, as scores = Q K^T (M = L, N = L, K = 128) or
    output = P V (M = L, N = 128, K = L), batch = heads; bf16 out,
    N(0, 1/sqrt(K)) inputs, seed 6000 + 100 * members + i."""
    seed = 6000 + 100 * members + i
    gen = torch.Generator(device="cpu")
    gen.manual_seed(seed)
    specs = []
    for _ in range(members):
        L = 128 * (1 << int(torch.randint(0, 5, (1,), generator=gen)[0]))
        heads = 16 * (1 + int(torch.randint(0, 2, (1,), generator=gen)[0]))
        if int(torch.randint(0, 2, (1,), generator=gen)[0]) == 0:
            M, N, K = L, L, 128
        else:
            M, N, K = L, 128, L
        specs.append(GemmSpec(M, N, K, DTYPE_BF16, "normal", 1.0 / math.sqrt(K), heads))
    return seed, specs


def make_batched_set(i: int, members: int) -> GemmSet:
    seed, specs = batched_study_specs(i, members)
    return materialize(f"bgemm{members}_{i:02d}", seed, specs)


def make_sweep_set(j: int) -> GemmSet:
    seed, specs, gen = sweep_specs(j)
    return materialize(f"sweep_{j:02d}", seed, specs, gen)


def random_matrix(rows: int, cols: int, seed: int, dist: str = "uniform",
                  scale: float = 1.0) -> torch.Tensor:
    """One seeded bf16 matrix (used for edge-case tests of odd shapes)."""
    gen = torch.Generator(device="cpu")
    gen.manual_seed(seed)
    return _draw(gen, rows, cols, dist, scale)


def integer_matrix(rows: int, cols: int, seed: int, lo: int = -8, hi: int = 8) -> torch.Tensor:
    """Seeded bf16 matrix of small integers in [lo, hi] (exact in bf16)."""
    gen = torch.Generator(device="cpu")
    gen.manual_seed(seed)
    x = torch.randint(lo, hi + 1, (rows, cols), generator=gen, dtype=torch.int32)
    return x.to(torch.float32).to(torch.bfloat16)
