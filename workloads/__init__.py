"""Seeded synthetic inputs for the CurvaDion step: layer-stack shapes, initial state, gradients.

This module only draws random numbers.  It holds none of the optimizer's arithmetic and
is shared by the tests, the benchmark and the oracle checks so that both sides of every
comparison receive identical inputs.  Every tensor comes from a ``torch.Generator`` on
the requested device seeded by (workload seed, layer, step), so a device-side draw is
reproducible and can be copied to the host for the oracle.

Workloads stand in for the paper's FineWeb GPT training runs (Section 4): the same
matrix shapes as its 160M / 350M / 1.3B GPT models, fp32 optimizer state, bf16
gradients (mixed-precision training), and gradient statistics chosen to exercise the
gate: i.i.d. Gaussian noise, a slowly rotating rank-8 component, and a rank-8 signal
whose scale alternates between flat and spiky phases.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import List, Tuple

import torch

# Gaussian parameters are given by their standard deviation.


@dataclass(frozen=True)
class Workload:
    name: str
    shapes: Tuple[Tuple[int, int], ...]  # (m, n) per layer, parameter X is m x n
    rank: int
    steps: int
    g_dtype: str  # "bf16" or "fp32"
    g_sigma: float
    kind: str = "gaussian"  # "gaussian" | "drift" | "spiky"
    x_sigma: float = 0.02
    seed: int = 0
    phase_len: int = 50  # spiky: steps per flat/spiky phase
    flat_scale: float = 0.1
    spiky_scale: float = 10.0
    drift_rad_per_step: float = 0.01
    drift_amp: float = 10.0  # drift amplitude = drift_amp * sigma * sqrt(max(m, n))
    signal_rank: int = 8

    @property
    def num_layers(self) -> int:
        return len(self.shapes)

    @property
    def elements(self) -> int:
        return sum(m * n for m, n in self.shapes)

    def ranks(self) -> List[int]:
        return [min(self.rank, m, n) for m, n in self.shapes]


def gpt_block(d: int, mlp: int) -> Tuple[Tuple[int, int], ...]:
    """The six Dion matrices of one GPT block: four d x d attention, d x mlp and mlp x d MLP."""
    return ((d, d),) * 4 + ((d, mlp), (mlp, d))


WORKLOADS = {
    # a single fp32 matrix, 10 steps
    "fp32_256x512_r16": Workload("fp32_256x512_r16", ((256, 512),), 16, 10, "fp32", 1e-2, seed=11),
    # one GPT-160M-shaped block (d = 768)
    "gpt160m_block_r192": Workload("gpt160m_block_r192", gpt_block(768, 3072), 192, 50, "bf16", 1e-3,
                                   seed=12),
    # full 160M-shaped stack: 12 blocks, 72 matrices, bf16 noise + rotating rank-8 component
    "gpt160m_stack_r192": Workload("gpt160m_stack_r192", gpt_block(768, 3072) * 12, 192, 100, "bf16",
                                   1e-3, kind="drift", seed=13),
    "gpt160m_stack_r48": Workload("gpt160m_stack_r48", gpt_block(768, 3072) * 12, 48, 100, "bf16",
                                  1e-3, kind="drift", seed=14),
    # 1.3B-shaped stack: 24 blocks, d = 2048, 144 matrices
    "gpt1p3b_stack_r512": Workload("gpt1p3b_stack_r512", gpt_block(2048, 8192) * 24, 512, 50, "bf16",
                                   1e-3, seed=15),
    # one block of the 1.3B-shaped stack (the profiling case: same shapes and rank, 6 matrices)
    "gpt1p3b_block_r512": Workload("gpt1p3b_block_r512", gpt_block(2048, 8192), 512, 50, "bf16", 1e-3, seed=15),
    # 350M-shaped gate stress stack: 24 blocks, d = 1024, flat/spiky phases every 50 steps
    "gpt350m_gate_stress_r256": Workload("gpt350m_gate_stress_r256", gpt_block(1024, 4096) * 24, 256,
                                         300, "bf16", 1e-3, kind="spiky", seed=16),
}


def _seed(w: Workload, layer: int, step: int, salt: int) -> int:
    return (w.seed * 1_000_003 + layer * 7_919 + step * 104_729 + salt * 15_485_863) & ((1 << 62) - 1)


def _gen(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def _randn(shape, device, seed, dtype=torch.float32):
    return torch.randn(shape, generator=_gen(device, seed), device=device, dtype=dtype)


def init_layer(w: Workload, layer: int, device="cpu"):
    """Initial (X_0, M_0, Q_0) of one layer.

    X_0 ~ N(0, x_sigma) fp32, M_0 = 0 (Algorithm 2's initialization), Q_0 = n x r Gaussian
    with every column scaled to unit length (a uniformly random direction per column).
    """
    m, n = w.shapes[layer]
    r = w.ranks()[layer]
    X = _randn((m, n), device, _seed(w, layer, 0, 1)) * w.x_sigma
    M = torch.zeros((m, n), device=device, dtype=torch.float32)
    q = _randn((n, r), device, _seed(w, layer, 0, 2), dtype=torch.float64)
    q = q / torch.linalg.vector_norm(q, dim=0, keepdim=True)
    return X.contiguous(), M, q.to(torch.float32).contiguous()


def _unit_columns(a: torch.Tensor) -> torch.Tensor:
    return a / torch.linalg.vector_norm(a, dim=0, keepdim=True)


def phase_scale(w: Workload, step: int) -> float:
    """Spiky workload: s_t = flat_scale in phases 0, 2, 4, ... and spiky_scale in phases 1, 3, ..."""
    phase = (step - 1) // w.phase_len
    return w.spiky_scale if phase % 2 == 1 else w.flat_scale


def gradient(w: Workload, layer: int, step: int, device="cpu") -> torch.Tensor:
    """G_t for one layer (step is the 1-based t), in the workload's gradient dtype."""
    m, n = w.shapes[layer]
    g = _randn((m, n), device, _seed(w, layer, step, 3)) * w.g_sigma
    k = w.signal_rank
    if w.kind == "drift":
        # rank-k component a * U(t) V(t)^T whose columns rotate in fixed random planes
        th = w.drift_rad_per_step * step
        a0 = _randn((m, k), device, _seed(w, layer, 0, 4))
        a1 = _randn((m, k), device, _seed(w, layer, 0, 5))
        c0 = _randn((n, k), device, _seed(w, layer, 0, 6))
        c1 = _randn((n, k), device, _seed(w, layer, 0, 7))
        u = _unit_columns(math.cos(th) * a0 + math.sin(th) * a1)
        v = _unit_columns(math.cos(th) * c0 + math.sin(th) * c1)
        amp = w.drift_amp * w.g_sigma * math.sqrt(max(m, n))
        g = g + amp * (u @ v.T)
    elif w.kind == "spiky":
        # fixed rank-k signal S with ||S||_F = sigma * sqrt(m n), scaled by the phase scale s_t
        u = _randn((m, k), device, _seed(w, layer, 0, 8))
        v = _randn((n, k), device, _seed(w, layer, 0, 9))
        s = u @ v.T
        s = s * (w.g_sigma * math.sqrt(m * n) / torch.linalg.vector_norm(s))
        g = g + phase_scale(w, step) * s
    elif w.kind != "gaussian":
        raise ValueError(w.kind)
    if w.g_dtype == "bf16":
        return g.to(torch.bfloat16).contiguous()
    if w.g_dtype == "fp32":
        return g.contiguous()
    raise ValueError(w.g_dtype)


def scaled(w: Workload, name: str, shapes, rank: int | None = None, steps: int | None = None,
           **kw) -> Workload:
    """A smaller variant of a workload (same statistics, other shapes) for oracle-sized tests."""
    fields = dict(w.__dict__)
    fields.update(name=name, shapes=tuple(tuple(s) for s in shapes))
    if rank is not None:
        fields["rank"] = rank
    if steps is not None:
        fields["steps"] = steps
    fields.update(kw)
    return Workload(**fields)


# ----------------------------------------------------------- quadratic objective (Theorem 1) ---
# Vector parameters (1 x n layers, rank 1) on F(x) = x^T H x / 2 with a symmetric positive
# definite H per layer whose eigenvalues are log-spaced in [lam_min, lam_max] and whose
# eigenvectors are a seeded random rotation.  The gradient H x is the test's input: it is
# computed from the parameters each step (a closed loop), with the same formula on both sides.

QUADRATIC_SHAPES = ((1, 1), (1, 64), (1, 512), (1, 2048))


def quadratic_hessian(n: int, seed: int, lam_min: float = 0.1, lam_max: float = 10.0, device="cpu") -> torch.Tensor:
    g = torch.Generator(device="cpu")
    g.manual_seed(seed)
    a = torch.randn((n, n), generator=g, dtype=torch.float64)
    u, _ = torch.linalg.qr(a)
    lam = torch.logspace(math.log10(lam_min), math.log10(lam_max), n, dtype=torch.float64)
    h = (u * lam[None, :]) @ u.T
    h = 0.5 * (h + h.T)
    return h.to(torch.float32).to(device)


def quadratic_start(n: int, seed: int, device="cpu") -> torch.Tensor:
    g = torch.Generator(device="cpu")
    g.manual_seed(seed)
    return torch.randn((1, n), generator=g, dtype=torch.float32).to(device)


def quadratic_gradient(H: torch.Tensor, X: torch.Tensor) -> torch.Tensor:
    """grad F = H x for a 1 x n row x (H symmetric): x H."""
    return X @ H
