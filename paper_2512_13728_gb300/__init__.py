"""GB300-native CurvaDion optimizer step (arXiv 2512.13728) behind a C ABI.

``native`` is the ctypes binding of include/curvadion.h (same names as the C entry points).
``Plan`` marshals torch CUDA tensors into ``dion_layer`` structs and owns the per-step
device outputs; torch is used only for device memory and streams.
"""
from __future__ import annotations

from typing import Optional, Sequence

from . import native
from .native import (DION_DTYPE_BF16, DION_DTYPE_FP32, DION_GATE_ALWAYS, DION_GATE_GLOBAL,  # noqa: F401
                     DION_GATE_PER_LAYER, DION_GATE_SCHEDULED, DION_PHASE_NORMS, DION_PHASE_ORTHO,
                     DION_PHASE_POWER, DION_PHASE_UPDATE, DION_PREC_BF16, DION_PREC_BF16X3,
                     DION_PREC_FP32, DionError, dion_hparams, dion_layer)


class _DeviceRange:
    """A plan-owned fp32 device range exposed through __cuda_array_interface__, so that
    torch.as_tensor views it without a copy (for a collective's in-place reduction)."""

    def __init__(self, ptr: int, count: int):
        self.__cuda_array_interface__ = {"shape": (count,), "typestr": "<f4", "data": (ptr, False), "version": 3}


def _layer(X, M, Q, G, tau: float) -> dion_layer:
    import torch

    for name, t in (("X", X), ("M", M), ("Q", Q)):
        if t.dtype != torch.float32 or not t.is_cuda or t.dim() != 2 or t.stride(1) != 1:
            raise ValueError(f"{name} must be a row-major 2-D float32 CUDA tensor")
    if G.dtype not in (torch.float32, torch.bfloat16) or not G.is_cuda or G.dim() != 2 or G.stride(1) != 1:
        raise ValueError("G must be a row-major 2-D float32 or bfloat16 CUDA tensor")
    m, n = X.shape
    r = Q.shape[1]
    if tuple(M.shape) != (m, n) or tuple(G.shape) != (m, n) or Q.shape[0] != n:
        raise ValueError("shape mismatch: X, M, G are m x n and Q is n x r")
    return dion_layer(m=m, n=n, r=r, X=X.data_ptr(), ldx=X.stride(0), M=M.data_ptr(), ldm=M.stride(0),
                      Q=Q.data_ptr(), ldq=Q.stride(0), G=G.data_ptr(), ldg=G.stride(0),
                      g_dtype=DION_DTYPE_BF16 if G.dtype == torch.bfloat16 else DION_DTYPE_FP32,
                      tau=float(tau))


def hparams(mu=0.95, eta=0.01, eta_local=None, eps_rmmc=1e-8, eps_col=1e-8, tau_global=0.5,
            gate_mode=DION_GATE_ALWAYS, period=1, step=1, weight_decay=0.0) -> dion_hparams:
    return dion_hparams(mu=mu, eta=eta, eta_local=eta if eta_local is None else eta_local, eps_rmmc=eps_rmmc,
                        eps_col=eps_col, tau_global=tau_global, gate_mode=gate_mode, period=period, step=step,
                        weight_decay=weight_decay)


def lr_schedule(step: int, total_steps: int, base_lr: float, warmup_frac: float = 0.01,
                warmdown_frac: float = 0.1) -> float:
    """Section 4's learning-rate schedule (the library's dion_lr_schedule)."""
    return native.dion_lr_schedule(step, total_steps, base_lr, warmup_frac, warmdown_frac)


def rank_for(m: int, n: int, fraction: float = 0.125) -> int:
    """Dion rank for a rank fraction (the library's dion_rank_for)."""
    return native.dion_rank_for(m, n, fraction)


class Plan:
    """A dion_plan over fixed torch tensors (X, M, Q, G per layer) plus device outputs.

    prev_norm (fp64 [L]) starts at 0 as Algorithm 2 initializes it; rmmc, rmmc_eq1 (fp64 [L]),
    flags (uint8 [L]) and global_flag (uint8 [1]) are rewritten by every step.
    """

    def __init__(self, X: Sequence, M: Sequence, Q: Sequence, G: Sequence, taus: Sequence[float],
                 precision: int = DION_PREC_FP32):
        import torch

        self._keep = (list(X), list(M), list(Q), list(G))
        self.layers = [_layer(x, m, q, g, t) for x, m, q, g, t in zip(X, M, Q, G, taus)]
        dev = X[0].device if len(X) else torch.device("cuda")
        L = len(self.layers)
        with torch.cuda.device(dev):
            self.handle = native.dion_plan_create(self.layers, precision)
        self.precision = precision
        self.device = dev
        self.prev_norm = torch.zeros(max(L, 1), dtype=torch.float64, device=dev)
        self.rmmc = torch.zeros(max(L, 1), dtype=torch.float64, device=dev)
        self.rmmc_eq1 = torch.zeros(max(L, 1), dtype=torch.float64, device=dev)
        self.flags = torch.zeros(max(L, 1), dtype=torch.uint8, device=dev)
        self.global_flag = torch.zeros(1, dtype=torch.uint8, device=dev)
        self.num_layers = L

    def step(self, hp: dion_hparams, stream: Optional[int] = None, eq1: bool = True) -> None:
        import torch

        s = torch.cuda.current_stream(self.device).cuda_stream if stream is None else stream
        native.dion_step(self.handle, hp, self.prev_norm.data_ptr(), self.rmmc.data_ptr(),
                         self.rmmc_eq1.data_ptr() if eq1 else None, self.flags.data_ptr(),
                         self.global_flag.data_ptr(), s)

    def step_phase(self, phase: int, hp: dion_hparams, stream: Optional[int] = None, eq1: bool = True) -> None:
        """One phase (DION_PHASE_*) of a data-parallel step; the caller reduces rmmc (max) after
        NORMS and the exchange() ranges (mean) after POWER and ORTHO."""
        import torch

        s = torch.cuda.current_stream(self.device).cuda_stream if stream is None else stream
        native.dion_step_phase(self.handle, phase, hp, self.prev_norm.data_ptr(), self.rmmc.data_ptr(),
                               self.rmmc_eq1.data_ptr() if eq1 else None, self.flags.data_ptr(),
                               self.global_flag.data_ptr(), s)

    def exchange(self, phase: int):
        """The plan's exchange range after `phase` (P after POWER, R after ORTHO) as a 1-D
        float32 tensor sharing the plan's memory (valid while the plan lives)."""
        import torch

        ptr, count = native.dion_plan_exchange(self.handle, phase)
        if count == 0:
            return torch.empty(0, dtype=torch.float32, device=self.device)
        return torch.as_tensor(_DeviceRange(ptr, count), device=self.device)

    def enable_host_gradients(self) -> None:
        """Lets step_host read each step's gradients from host memory (two device buffers per
        layer, filled in turn on the plan's copy stream)."""
        native.dion_plan_enable_host_gradients(self.handle)

    def step_host(self, hp: dion_hparams, host_G: Sequence, stream: Optional[int] = None, eq1: bool = True) -> None:
        """One step with the gradients read from host tensors (row-major 2-D CPU tensors of each
        layer's gradient dtype and shape; pinned memory lets the copies overlap the previous
        step).  The tensors must not change until the step's stream has passed its start."""
        import torch

        if len(host_G) != self.num_layers:
            raise ValueError("one host gradient per layer")
        for g, ly in zip(host_G, self.layers):
            want = torch.bfloat16 if ly.g_dtype == DION_DTYPE_BF16 else torch.float32
            if g.is_cuda or g.dtype != want or g.dim() != 2 or tuple(g.shape) != (ly.m, ly.n) or g.stride(1) != 1:
                raise ValueError("host gradients must be row-major CPU tensors of the layer's shape and dtype")
        s = torch.cuda.current_stream(self.device).cuda_stream if stream is None else stream
        native.dion_step_host(self.handle, hp, [g.data_ptr() for g in host_G], [g.stride(0) for g in host_G],
                              self.prev_norm.data_ptr(), self.rmmc.data_ptr(),
                              self.rmmc_eq1.data_ptr() if eq1 else None, self.flags.data_ptr(),
                              self.global_flag.data_ptr(), s)

    def refresh(self, stream: Optional[int] = None) -> None:
        """Call after writing Q from outside dion_step (e.g. a checkpoint restore)."""
        import torch

        s = torch.cuda.current_stream(self.device).cuda_stream if stream is None else stream
        native.dion_plan_refresh(self.handle, s)

    def device_status(self, clear: bool = True) -> int:
        return native.dion_get_device_status(self.handle, clear)

    def check_guards(self) -> int:
        """Damaged workspace guard words (synchronizes the device)."""
        return native.dion_plan_check_guards(self.handle)

    def launches_per_step(self) -> int:
        return native.dion_step_launch_count(self.handle)

    def close(self) -> None:
        if getattr(self, "handle", None):
            native.dion_plan_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
