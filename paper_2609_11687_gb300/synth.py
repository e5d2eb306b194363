"""Seeded synthetic weight matrices shaped like the paper's models.

The paper evaluates on trained OPT, Llama-2, Pythia and Mistral weights (Sec. 4);
none are available here, so every workload is a seeded random stand-in with the
layer shapes of those models.  This module only draws random numbers: it holds
none of the decomposition's arithmetic and is the one module that both the CPU
oracle's tests and the CUDA path's tests/bench import.

Conventions
-----------
The paper writes a layer as ``W in R^{N x M}`` (N input features, M output
channels) and decomposes every column ``W[:, j]`` (App. C).  Generators here
return the *vector-major* tensor ``G`` of shape ``(M, N)`` with ``G[j] = W[:, j]``
-- the ``nn.Linear.weight`` layout ``[out, in]`` -- so each decomposed vector is a
contiguous row of ``G``.

Distributions (all from one ``torch.Generator`` seeded per matrix):

* ``normal``   : ``std * Z``.
* ``student_t``: ``t_nu = Z_0 / sqrt(sum_{i=1..nu} Z_i^2 / nu)``, rescaled to the
  requested standard deviation (``Var t_nu = nu / (nu - 2)``).
* outlier input channels: ``round(frac * N)`` positions along N drawn with
  ``randperm`` are multiplied by ``scale`` in every vector.
* outlier entries: ``round(frac * M * N)`` flat positions drawn with ``randint``
  are multiplied by ``scale``.
"""

from __future__ import annotations

import dataclasses
import math
from typing import Iterator, List, Sequence, Tuple

import torch


@dataclasses.dataclass(frozen=True)
class MatrixSpec:
    """One synthetic weight matrix: ``N`` = vector length, ``M`` = number of vectors."""

    name: str
    N: int
    M: int
    seed: int
    dist: str = "student_t"  # "normal" | "student_t"
    nu: int = 4
    std: float = 0.02
    dtype: torch.dtype = torch.float16
    outlier_channel_frac: float = 0.0
    outlier_channel_scale: float = 1.0
    outlier_entry_frac: float = 0.0
    outlier_entry_scale: float = 1.0

    @property
    def sign_seed(self) -> int:
        return self.seed

    @property
    def params(self) -> int:
        return self.N * self.M


def generate(spec: MatrixSpec, device: str | torch.device = "cpu") -> torch.Tensor:
    """Draw ``spec`` as an ``(M, N)`` tensor of ``spec.dtype`` on ``device``.

    The same (spec, device type) always gives the same bits; CPU and CUDA
    generators are different streams, so a test that compares against the
    oracle must copy the values it uses from the device that drew them.
    """
    dev = torch.device(device)
    g = torch.Generator(device=dev)
    g.manual_seed(int(spec.seed))
    shape = (spec.M, spec.N)
    if spec.dist == "normal":
        x = torch.randn(shape, generator=g, device=dev, dtype=torch.float32) * spec.std
    elif spec.dist == "student_t":
        nu = int(spec.nu)
        z0 = torch.randn(shape, generator=g, device=dev, dtype=torch.float32)
        acc = torch.zeros(shape, device=dev, dtype=torch.float32)
        for _ in range(nu):
            zi = torch.randn(shape, generator=g, device=dev, dtype=torch.float32)
            acc.addcmul_(zi, zi)
        x = z0 / torch.sqrt(acc / nu)
        x.mul_(spec.std / math.sqrt(nu / (nu - 2.0)))
    else:
        raise ValueError(f"unknown distribution {spec.dist!r}")
    if spec.outlier_channel_frac > 0.0:
        n_out = int(round(spec.outlier_channel_frac * spec.N))
        if n_out > 0:
            idx = torch.randperm(spec.N, generator=g, device=dev)[:n_out]
            x[:, idx] *= spec.outlier_channel_scale
    if spec.outlier_entry_frac > 0.0:
        n_out = int(round(spec.outlier_entry_frac * spec.M * spec.N))
        if n_out > 0:
            flat = torch.randint(0, spec.M * spec.N, (n_out,), generator=g, device=dev)
            xv = x.view(-1)
            xv[flat] = xv[flat] * spec.outlier_entry_scale
    return x.to(spec.dtype)


# ---------------------------------------------------------------------------
# Workload recipes (the five configurations).  Shapes are (N in, M out).
# ---------------------------------------------------------------------------

def config1() -> List[MatrixSpec]:
    """Single 256x256 fp32 matrix, entries 0.02 * N(0, 1), seed 0."""
    return [MatrixSpec("w256", 256, 256, seed=0, dist="normal", std=0.02, dtype=torch.float32)]


_OPT125M = [("q", 768, 768), ("k", 768, 768), ("v", 768, 768), ("o", 768, 768),
            ("fc1", 768, 3072), ("fc2", 3072, 768)]


def config2(layers: Sequence[int] = range(12)) -> List[MatrixSpec]:
    """OPT-125M-shaped layer set, fp16, Student-t nu=4 scaled to std 0.02."""
    out = []
    for layer in layers:
        for mi, (nm, n, m) in enumerate(_OPT125M):
            out.append(MatrixSpec(f"L{layer}.{nm}", n, m, seed=1000 * layer + mi,
                                  dist="student_t", nu=4, std=0.02))
    return out


_LLAMA7B = [("q", 4096, 4096), ("k", 4096, 4096), ("v", 4096, 4096), ("o", 4096, 4096),
            ("gate", 4096, 11008), ("up", 4096, 11008), ("down", 11008, 4096)]


def llama7b_layer(layer: int) -> List[MatrixSpec]:
    """One Llama-2-7B-shaped decoder layer: Student-t nu=4, std 0.015, 0.1% of
    input channels scaled x20."""
    return [MatrixSpec(f"L{layer}.{nm}", n, m, seed=1000 * layer + mi, dist="student_t", nu=4,
                       std=0.015, outlier_channel_frac=0.001, outlier_channel_scale=20.0)
            for mi, (nm, n, m) in enumerate(_LLAMA7B)]


def config3() -> List[MatrixSpec]:
    return llama7b_layer(0)


def config4(layers: Sequence[int] = range(32)) -> List[MatrixSpec]:
    out = []
    for layer in layers:
        out.extend(llama7b_layer(layer))
    return out


_PYTHIA69B = [("qkv", 4096, 12288), ("dense", 4096, 4096), ("h_4h", 4096, 16384), ("4h_h", 16384, 4096)]
_MISTRAL7B = [("q", 4096, 4096), ("k", 4096, 1024), ("v", 4096, 1024), ("o", 4096, 4096),
              ("gate", 4096, 14336), ("up", 4096, 14336), ("down", 14336, 4096)]


def config5(layers: Sequence[int] = range(32)) -> List[MatrixSpec]:
    """Stress shapes: Student-t nu=3 (std 0.02 before outliers), 0.05% entries x50."""
    out = []
    for fam, shapes, base in (("pythia", _PYTHIA69B, 100000), ("mistral", _MISTRAL7B, 200000)):
        for layer in layers:
            for mi, (nm, n, m) in enumerate(shapes):
                out.append(MatrixSpec(f"{fam}.L{layer}.{nm}", n, m, seed=base + 1000 * layer + mi,
                                      dist="student_t", nu=3, std=0.02,
                                      outlier_entry_frac=0.0005, outlier_entry_scale=50.0))
    return out


def gaussian_vectors(n: int, m: int = 1, seed: int = 0) -> MatrixSpec:
    """Fig. 2's input: ``m`` vectors of length ``n`` drawn from N(0, I_n), fp32."""
    return MatrixSpec(f"gauss{n}x{m}", n, m, seed=seed, dist="normal", std=1.0, dtype=torch.float32)


CONFIGS = {1: config1, 2: config2, 3: config3, 4: config4, 5: config5}


def total_params(specs: Sequence[MatrixSpec]) -> int:
    return sum(s.params for s in specs)


def pair_aligned_sample(M: int, n_vectors: int, seed: int) -> List[int]:
    """Seeded sample of vector indices that keeps the (2j, 2j+1) pairs whole.

    The GPU path processes vectors two at a time, so a sampled vector is always
    taken together with its neighbour; returns sorted indices.
    """
    n_pairs_total = (M + 1) // 2
    n_pairs = max(1, min(n_pairs_total, (n_vectors + 1) // 2))
    g = torch.Generator().manual_seed(int(seed))
    pairs = torch.randperm(n_pairs_total, generator=g)[:n_pairs].sort().values.tolist()
    out = []
    for p in pairs:
        out.append(2 * p)
        if 2 * p + 1 < M:
            out.append(2 * p + 1)
    return out
