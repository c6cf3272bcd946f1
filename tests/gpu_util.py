"""Helpers of the GPU parity tests: build device state from a workload, snapshot it for the
oracle, run one library step and one oracle step from the same state, compare."""
from __future__ import annotations

import math
from dataclasses import dataclass
from typing import List, Optional

import numpy as np
import torch

import oracle.curvadion as oc
import workloads as wl


def f32(x: float) -> float:
    """The fp32 value the library sees for a hyper-parameter, widened back to fp64."""
    return float(np.float32(x))


def rel_fro(got, want) -> float:
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    den = np.linalg.norm(want)
    return float(np.linalg.norm(got - want) / (den if den > 0 else 1.0))


@dataclass
class DevState:
    w: wl.Workload
    X: List[torch.Tensor]
    M: List[torch.Tensor]
    Q: List[torch.Tensor]
    G: List[torch.Tensor]
    taus: List[float]


def make_state(w: wl.Workload, device="cuda", taus: Optional[List[float]] = None, pad: int = 0) -> DevState:
    """Initial state of workload w on the device.  Every tensor's leading dimension is its width
    rounded up to a multiple of 8 elements (16-byte rows), plus 8 * pad; padding holds NaN so
    that a kernel reading past a row's end would poison the result."""
    X, M, Q, G = [], [], [], []
    gdt = torch.bfloat16 if w.g_dtype == "bf16" else torch.float32
    for l, (m, n) in enumerate(w.shapes):
        x0, m0, q0 = wl.init_layer(w, l, device)
        r = q0.shape[1]

        def padded(t, cols, dtype=torch.float32):
            # rows 16-byte aligned for both fp32 and bf16: leading dimension a multiple of 8
            ld = (cols + 7) // 8 * 8 + 8 * pad
            if ld == cols:
                return t.contiguous()
            buf = torch.full((t.shape[0], ld), float("nan"), device=device, dtype=dtype)
            buf[:, :cols] = t
            return buf[:, :cols]

        X.append(padded(x0, n))
        M.append(padded(m0, n))
        Q.append(padded(q0, r))
        G.append(padded(torch.zeros((m, n), device=device, dtype=gdt), n, gdt))
    taus = list(taus) if taus is not None else [0.5] * w.num_layers
    return DevState(w, X, M, Q, G, taus)


def write_gradients(st: DevState, step: int):
    for l in range(st.w.num_layers):
        st.G[l].copy_(wl.gradient(st.w, l, step, st.G[l].device))


def snapshot(st: DevState, plan=None):
    """Host fp64 copies of the state (what the oracle takes) and of this step's gradients."""
    layers = [oc.LayerState(X=oc.as_f64(st.X[l]), M=oc.as_f64(st.M[l]), Q=oc.as_f64(st.Q[l]), tau=f32(st.taus[l]))
              for l in range(st.w.num_layers)]
    grads = [oc.as_f64(st.G[l]) for l in range(st.w.num_layers)]
    prev = plan.prev_norm[: st.w.num_layers].double().cpu().numpy().copy() if plan is not None else None
    return layers, grads, prev


def oracle_hp(mu=0.95, eta=0.01, eta_local=None, eps_rmmc=1e-8, eps_col=1e-8, tau_global=0.5, gate_mode=0,
              period=1, weight_decay=0.0) -> oc.HParams:
    return oc.HParams(mu=f32(mu), eta=f32(eta), eta_local=f32(eta if eta_local is None else eta_local),
                      eps_rmmc=f32(eps_rmmc), eps_col=f32(eps_col), gate_mode=gate_mode, tau_global=f32(tau_global),
                      period=period, weight_decay=f32(weight_decay))


@dataclass
class StepCompare:
    err_M: float
    err_X: float
    err_Q: float
    err_rmmc: float
    err_eq1: float
    flags_equal: bool
    gflag_equal: bool
    margin: float  # min over layers of |RMMC - tau| / tau (near-tie indicator)
    want: oc.StepOutput


def compare_step(st: DevState, plan, layers, grads, prev, hp: oc.HParams, step: int, layer_ids=None) -> StepCompare:
    """Oracle step from the snapshot (layers, grads, prev) vs the device state after the library's step."""
    L = st.w.num_layers
    want = oc.curvadion_step(layers, grads, prev, hp, step)
    ids = range(L) if layer_ids is None else layer_ids
    eM = max(rel_fro(oc.as_f64(st.M[l]), want.layers[l].M) for l in ids)
    eX = max(rel_fro(oc.as_f64(st.X[l]), want.layers[l].X) for l in ids)
    eQ = max(rel_fro(oc.as_f64(st.Q[l]), want.layers[l].Q) for l in ids)
    rm = plan.rmmc[:L].double().cpu().numpy()
    eq1 = plan.rmmc_eq1[:L].double().cpu().numpy()
    flags = plan.flags[:L].cpu().numpy().astype(bool)
    gflag = bool(plan.global_flag[0].item())
    # relative error, absolute below 1 (norms carry ~1e-7 relative error from fp32 partial sums)
    finite = np.isfinite(want.rmmc)
    err_rm = float(np.max(np.abs(rm[finite] - want.rmmc[finite]) / np.maximum(np.abs(want.rmmc[finite]), 1.0))) \
        if finite.any() else 0.0
    err_eq1 = float(np.max(np.abs(eq1 - want.rmmc_eq1) / np.maximum(np.abs(want.rmmc_eq1), 1.0))) if L else 0.0
    taus = np.array([lay.tau for lay in layers])
    margin = float(np.min(np.abs(want.rmmc - taus) / np.maximum(np.abs(taus), 1e-30))) if L else math.inf
    return StepCompare(eM, eX, eQ, err_rm, err_eq1, bool(np.array_equal(flags, want.flags)),
                       gflag == want.global_flag, margin, want)
