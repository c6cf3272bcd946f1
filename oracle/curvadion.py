"""fp64 CPU oracle of one CurvaDion optimizer step (arXiv 2512.13728).

TEST INFRASTRUCTURE ONLY.  This module is the slow, obviously-correct reference that the
GPU path is checked against.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import it.  It shares no
code with the CUDA library and imports nothing from it.

Everything is float64 numpy.  Inputs given in fp32 or bf16 are widened exactly.  Each
function names the passage of the paper it follows:

* Algorithm 1 (Dion baseline): buffer, power iteration, orthogonalize, error feedback,
  column normalization, scaled low-rank parameter update.
* Algorithm 2 (CurvaDion): per-layer RMMC with prev_norm and epsilon, max over layers,
  strict threshold compare, sync branch = the Dion update, local branch = M <- B, X -= eta_local G.
* Equation 1: RMMC from the momentum norms of consecutive steps (reported as a diagnostic).

Readings where the paper is silent (each is also listed in the design notes):

* the norm is the Frobenius norm (the proof of Theorem 1 expands ||M_t||^2 as an inner product);
* R is computed from the orthonormalized P, after Orthogonalize (Algorithm 1 lists P and R
  as one power-iteration output but reduces R after the orthogonalization);
* Orthogonalize returns the Q factor of the thin QR of P whose triangular factor has a
  positive diagonal (unique for full-rank P);
* ColumnNormalize divides each column by (its 2-norm + eps_col);
* sqrt(m/n) uses m = rows, n = columns of the parameter matrix X;
* a non-finite RMMC counts as above every threshold;
* Equation 1's ratio takes the same epsilon as Algorithm 2 in its denominator so that the
  first step (zero momentum) is finite;
* the local branch keeps M = B with no decay, exactly as Algorithm 2 writes it.
* weight decay (Section 4 trains with 0.01 but Algorithms 1/2 have no such line) is decoupled:
  X is multiplied by (1 - lr * weight_decay) before the branch's update, lr being the branch's
  learning rate (eta for the Dion update, eta_local for the local one); weight_decay = 0 is the
  algorithm as printed;
* the learning-rate schedule (Section 4: 1% warmup, 10% or 20% warmdown) is linear: it rises
  from base/W at step 1 to base at step W, stays at base, and falls linearly to 0 at the last
  step over the final D steps (W, D = warmup_frac * T, warmdown_frac * T rounded half up);
* the Dion rank for a rank fraction f (Section 4: f = 0.125) is ceil(f * min(m, n)), at least 1.

Pins: ``tests/test_oracle_pins.py`` checks every function here against results fixed by
the paper or by mathematics (closed forms, LAPACK, brute force on tiny cases).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import List, Optional, Sequence

import numpy as np

# Gate modes.  ALWAYS is Algorithm 1 (every step synchronizes; RMMC only reported).
# GLOBAL is Algorithm 2 (one decision from the max over layers).  PER_LAYER thresholds
# each layer's own RMMC.  SCHEDULED is the Scheduled Sync Dion baseline of Section 4.3 and Appendix C:
# synchronize on every H-th step, local updates otherwise.
GATE_ALWAYS = 0
GATE_GLOBAL = 1
GATE_PER_LAYER = 2
GATE_SCHEDULED = 3


def as_f64(a) -> np.ndarray:
    """Widen an fp32/bf16/fp64 array-like (numpy or torch CPU tensor) to float64 exactly."""
    if hasattr(a, "detach"):  # torch tensor: bf16 has no numpy dtype, widen through float32
        import torch  # local import: plain torch CPU ops only

        t = a.detach().cpu()
        if t.dtype == torch.bfloat16:
            t = t.to(torch.float32)
        return t.to(torch.float64).numpy().copy()
    return np.asarray(a, dtype=np.float64).copy()


# ---------------------------------------------------------------------------------------
# Algorithm 1 / Algorithm 2 building blocks
# ---------------------------------------------------------------------------------------

def form_buffer(M: np.ndarray, G: np.ndarray) -> np.ndarray:
    """B_t = M_{t-1} + G_t (Algorithm 1 and Algorithm 2, 'update buffer')."""
    return M + G


def frobenius_norm(A: np.ndarray) -> float:
    """||A|| read as the Frobenius norm: the square root of the sum of squared entries."""
    return math.sqrt(float(np.sum(A * A)))


def rmmc_alg2(norm_b: float, prev_norm: float, eps: float) -> float:
    """Algorithm 2's per-layer RMMC: | ||B_t|| - prev_norm | / (prev_norm + eps)."""
    return abs(norm_b - prev_norm) / (prev_norm + eps)


def rmmc_eq1(norm_now: float, norm_before: float, eps: float) -> float:
    """Equation 1: | ||M(t)|| - ||M(t-1)|| | / ||M(t-1)||, with eps added to the denominator."""
    return abs(norm_now - norm_before) / (norm_before + eps)


def power_iter(B: np.ndarray, Q_prev: np.ndarray) -> np.ndarray:
    """PowerIter (Algorithm 1): one multiplication of the buffer by the previous right factor, P = B Q_{t-1}."""
    return B @ Q_prev


def householder_qr(A: np.ndarray):
    """Thin QR of an m x r matrix (m >= r) by Householder reflections.

    Returns (Qf, Rf) with A = Qf Rf, Qf^T Qf = I_r and diag(Rf) >= 0.  This is the
    Orthogonalize step of Algorithm 1/2 under the positive-diagonal reading.
    Textbook algorithm: column j is reflected onto a multiple of e_j by
    H_j = I - 2 v v^T, with v chosen to avoid cancellation; the Q factor is
    H_0 H_1 ... H_{r-1} applied to the first r columns of the identity.
    """
    W = np.array(A, dtype=np.float64, copy=True)
    m, r = W.shape
    if r > m:
        raise ValueError("householder_qr needs m >= r")
    vs = []
    for j in range(r):
        x = W[j:, j]
        nx = math.sqrt(float(x @ x))
        v = x.copy()
        if nx == 0.0:
            vs.append(None)  # column already zero below the diagonal: H_j = I
            continue
        alpha = -nx if x[0] >= 0.0 else nx
        v[0] -= alpha
        nv = math.sqrt(float(v @ v))
        if nv == 0.0:
            vs.append(None)
            continue
        v /= nv
        W[j:, j:] -= 2.0 * np.outer(v, v @ W[j:, j:])
        vs.append(v)
    Rf = np.triu(W[:r, :r])
    Qf = np.zeros((m, r))
    Qf[:r, :r] = np.eye(r)
    for j in reversed(range(r)):
        v = vs[j]
        if v is None:
            continue
        Qf[j:, :] -= 2.0 * np.outer(v, v @ Qf[j:, :])
    # Positive-diagonal convention: flip column j of Q and row j of R where R_jj < 0.
    d = np.where(np.diag(Rf) < 0.0, -1.0, 1.0)
    return Qf * d[None, :], Rf * d[:, None]


def orthogonalize(P: np.ndarray) -> np.ndarray:
    """Orthogonalize(P) (Algorithm 1/2): the orthonormal Q factor of the thin QR of P."""
    return householder_qr(P)[0]


def column_normalize(R: np.ndarray, eps_col: float) -> np.ndarray:
    """ColumnNormalize(R) (Algorithm 1/2): column j divided by (||R[:, j]||_2 + eps_col)."""
    norms = np.sqrt(np.sum(R * R, axis=0))
    return R / (norms[None, :] + eps_col)


@dataclass
class SyncResult:
    M: np.ndarray
    Q: np.ndarray
    X: np.ndarray
    P: np.ndarray
    R: np.ndarray


def decay_parameters(X, lr: float, weight_decay: float):
    """Decoupled weight decay applied before a branch's update: (1 - lr * weight_decay) X."""
    return (1.0 - lr * weight_decay) * X


def lr_schedule(step: int, total_steps: int, base_lr: float, warmup_frac: float, warmdown_frac: float) -> float:
    """Learning rate at 1-based ``step`` of a ``total_steps`` run (Section 4's warmup/warmdown).

    W = warmup_frac * T and D = warmdown_frac * T, each rounded half up, must fit in T.
    W warmup steps: base * step / W for step <= W.  D warmdown steps: base * (T - step) / D for
    step > T - D (ending at 0 on the last step).  Otherwise base.  Steps outside [1, T] clamp.
    """
    T = int(total_steps)
    t = min(max(int(step), 1), T)
    W = int(math.floor(warmup_frac * T + 0.5))
    D = int(math.floor(warmdown_frac * T + 0.5))
    if T < 1 or W + D > T:
        raise ValueError("warmup and warmdown do not fit in the run")
    if W > 0 and t <= W:
        return base_lr * t / W
    if D > 0 and t > T - D:
        return base_lr * (T - t) / D
    return base_lr


def rank_for(m: int, n: int, fraction: float) -> int:
    """Dion rank from a rank fraction (Section 4: r = 0.125): ceil(fraction * min(m, n)), >= 1."""
    k = min(m, n)
    return max(1, min(k, int(math.ceil(fraction * k - 1e-12))))


def dion_sync_update(B, Q_prev, X, mu: float, eta: float, eps_col: float, weight_decay: float = 0.0) -> SyncResult:
    """The synchronized branch of Algorithm 2 (= one step of Algorithm 1 after the buffer).

    With one data-parallel worker the two AllReduce_DP lines are the identity.
      P  = PowerIter(B; Q_{t-1}) = B Q_{t-1}
      P  = Orthogonalize(P)
      R  = B^T P
      M  = B - (1 - mu) P R^T
      Q  = ColumnNormalize(R)
      X  = X - eta sqrt(m/n) P Q^T      (after decoupled weight decay of X, if any)
    """
    m, n = B.shape
    P = orthogonalize(power_iter(B, Q_prev))
    R = B.T @ P
    M_new = B - (1.0 - mu) * (P @ R.T)
    Q_new = column_normalize(R, eps_col)
    X_new = decay_parameters(X, eta, weight_decay) - eta * math.sqrt(m / n) * (P @ Q_new.T)
    return SyncResult(M=M_new, Q=Q_new, X=X_new, P=P, R=R)


def local_update(B, G, X, eta_local: float, weight_decay: float = 0.0):
    """The local branch of Algorithm 2: M = B (no decay) and X = X - eta_local G (after
    decoupled weight decay of X, if any)."""
    return B.copy(), decay_parameters(X, eta_local, weight_decay) - eta_local * G


# ---------------------------------------------------------------------------------------
# The gate (Algorithm 2) and a whole multi-layer step
# ---------------------------------------------------------------------------------------

def above(value: float, tau: float) -> bool:
    """Strict threshold compare of Algorithm 2 ('> tau'); a non-finite RMMC is above every tau."""
    return (not math.isfinite(value)) or value > tau


def gate(rmmc: Sequence[float], taus: Sequence[float], tau_global: float, mode: int,
         step: int, period: int):
    """Sync decisions for one step.

    Returns (flags, global_flag, active): flags[l] = RMMC_l > tau_l, global_flag = max_l RMMC_l > tau_global
    (Algorithm 2's AllReduce_max over one worker is the max over layers), and active[l] says
    which layers take the Dion branch under ``mode``.
    """
    L = len(rmmc)
    flags = [above(rmmc[i], taus[i]) for i in range(L)]
    gmax = -math.inf
    for v in rmmc:
        gmax = math.inf if not math.isfinite(v) else max(gmax, v)
    global_flag = above(gmax, tau_global) if L > 0 else False
    if mode == GATE_ALWAYS:
        active = [True] * L
    elif mode == GATE_GLOBAL:
        active = [global_flag] * L
    elif mode == GATE_PER_LAYER:
        active = list(flags)
    elif mode == GATE_SCHEDULED:
        if period < 1:
            raise ValueError("scheduled gate needs period >= 1")
        active = [step % period == 0] * L
    else:
        raise ValueError(f"unknown gate mode {mode}")
    return flags, global_flag, active


@dataclass
class LayerState:
    X: np.ndarray  # m x n parameters
    M: np.ndarray  # m x n momentum
    Q: np.ndarray  # n x r right factor
    tau: float = 0.5


@dataclass
class HParams:
    mu: float = 0.95
    eta: float = 0.01
    eta_local: float = 0.01
    eps_rmmc: float = 1e-8
    eps_col: float = 1e-8
    gate_mode: int = GATE_ALWAYS
    tau_global: float = 0.5
    period: int = 1
    weight_decay: float = 0.0


@dataclass
class StepOutput:
    layers: List[LayerState]
    prev_norm: np.ndarray
    rmmc: np.ndarray
    rmmc_eq1: np.ndarray
    flags: np.ndarray
    global_flag: bool
    active: np.ndarray
    norm_b: np.ndarray
    extras: list = field(default_factory=list)


def curvadion_step(layers: Sequence[LayerState], grads: Sequence[np.ndarray],
                   prev_norm: Sequence[float], hp: HParams, step: int,
                   keep_extras: bool = False) -> StepOutput:
    """One step of Algorithm 2 over all layers (Algorithm 1 when hp.gate_mode == GATE_ALWAYS).

    ``step`` is the 1-based t.  Inputs are not modified.  The returned prev_norm holds
    ||B_t|| per layer, as Algorithm 2 assigns it.
    """
    L = len(layers)
    Bs, nb, rm = [], np.zeros(L), np.zeros(L)
    norm_m_before = np.zeros(L)
    for i, (st, G) in enumerate(zip(layers, grads)):
        M = as_f64(st.M)
        norm_m_before[i] = frobenius_norm(M)
        B = form_buffer(M, as_f64(G))
        Bs.append(B)
        nb[i] = frobenius_norm(B)
        rm[i] = rmmc_alg2(nb[i], float(prev_norm[i]), hp.eps_rmmc)
    flags, gflag, active = gate(rm, [st.tau for st in layers], hp.tau_global, hp.gate_mode,
                                step, hp.period)
    out_layers, eq1, extras = [], np.zeros(L), []
    for i, st in enumerate(layers):
        X = as_f64(st.X)
        if active[i]:
            res = dion_sync_update(Bs[i], as_f64(st.Q), X, hp.mu, hp.eta, hp.eps_col, hp.weight_decay)
            new = LayerState(X=res.X, M=res.M, Q=res.Q, tau=st.tau)
            if keep_extras:
                extras.append(res)
        else:
            M_new, X_new = local_update(Bs[i], as_f64(grads[i]), X, hp.eta_local, hp.weight_decay)
            new = LayerState(X=X_new, M=M_new, Q=as_f64(st.Q), tau=st.tau)
            if keep_extras:
                extras.append(None)
        eq1[i] = rmmc_eq1(frobenius_norm(new.M), norm_m_before[i], hp.eps_rmmc)
        out_layers.append(new)
    return StepOutput(layers=out_layers, prev_norm=nb.copy(), rmmc=rm, rmmc_eq1=eq1,
                      flags=np.array(flags, dtype=bool), global_flag=bool(gflag),
                      active=np.array(active, dtype=bool), norm_b=nb, extras=extras)


def run_trajectory(layers: Sequence[LayerState], grad_fn, steps: int, hp: HParams,
                   prev_norm: Optional[Sequence[float]] = None):
    """Run ``steps`` steps from t = 1 (Algorithm 2's loop); grad_fn(layer, t) gives G_t.

    prev_norm starts at 0 for every layer (Algorithm 2's initialization).
    Returns (final layers, list of StepOutput).
    """
    cur = list(layers)
    pn = np.zeros(len(cur)) if prev_norm is None else np.asarray(prev_norm, dtype=np.float64)
    outs = []
    for t in range(1, steps + 1):
        o = curvadion_step(cur, [grad_fn(i, t) for i in range(len(cur))], pn, hp, t)
        outs.append(o)
        cur, pn = o.layers, o.prev_norm
    return cur, outs


# ---------------------------------------------------------------------------------------
# Theorem 1 (RMMC and directional curvature) on a quadratic objective
# ---------------------------------------------------------------------------------------
# For a 1 x n parameter the Dion branch is heavy-ball momentum with a normalized step: r = 1,
# P = sign(B Q_{t-1}) (1 x 1), R = B^T P, Q_t = R / (||R|| + eps_col), so
#   X_t = X_{t-1} - eta sqrt(1/n) B / (||B|| + eps_col)   and   M_t = mu B,
# i.e. B_t = mu B_{t-1} + G_t is the theorem's momentum M_t and the step is x_t = x_{t-1} -
# eta_eff M_{t-1} with eta_eff = eta / (sqrt(n) (||B_{t-1}|| + eps_col)).  On F(x) = x^T H x / 2
# the gradient expansion of the proof is exact, so with v = B_{t-1} / ||B_{t-1}||,
# kappa = v^T H v, B_t = (1 - mu) - v^T grad F(x_{t-1}) / ||B_{t-1}||, and rho = the part of
# grad F(x_t) perpendicular to v divided by ||B_{t-1}||:
#   ||B_t|| / ||B_{t-1}|| = sqrt((1 - B_t - eta_eff kappa)^2 + rho^2),
# which is Theorem 1's |eta kappa + B_t| when rho = 0 (exactly so for n = 1); otherwise the
# two differ by at most rho^2 / (2 (1 - B_t - eta_eff kappa)) (sqrt(a^2 + c) - a <= c / (2a)).

def rank1_step_size(eta: float, n: int, b_prev: np.ndarray, eps_col: float) -> float:
    """eta_eff of a 1 x n layer's Dion step: eta / (sqrt(n) (||B_{t-1}|| + eps_col))."""
    return eta / (math.sqrt(n) * (frobenius_norm(b_prev) + eps_col))


@dataclass
class Theorem1Terms:
    kappa: float        # v^T H v, v = B_{t-1} / ||B_{t-1}||
    bias: float         # B_t = (1 - mu) - v^T grad F(x_{t-1}) / ||B_{t-1}||
    eta_eff: float
    prediction: float   # |eta_eff kappa + B_t|
    rho: float          # |grad F(x_t) perpendicular to v| / ||B_{t-1}||
    exact: float        # |sqrt((1 - B_t - eta_eff kappa)^2 + rho^2) - 1|


def theorem1_terms(H: np.ndarray, x_prev: np.ndarray, b_prev: np.ndarray, mu: float, eta_eff: float) -> Theorem1Terms:
    """Theorem 1's quantities for the step from x_{t-1} (1 x n) with momentum B_{t-1} on
    F(x) = x^T H x / 2 (H symmetric), and the exact ratio of the momentum norms."""
    H = as_f64(H)
    x_prev = as_f64(x_prev).reshape(-1)
    b_prev = as_f64(b_prev).reshape(-1)
    m_prev = float(np.linalg.norm(b_prev))
    v = b_prev / m_prev
    g_prev = H @ x_prev
    kappa = float(v @ H @ v)
    bias = (1.0 - mu) - float(v @ g_prev) / m_prev
    x_now = x_prev - eta_eff * b_prev
    g_now = H @ x_now
    g_perp = g_now - float(v @ g_now) * v
    rho = float(np.linalg.norm(g_perp)) / m_prev
    a = 1.0 - bias - eta_eff * kappa
    return Theorem1Terms(kappa=kappa, bias=bias, eta_eff=eta_eff, prediction=abs(eta_eff * kappa + bias),
                         rho=rho, exact=abs(math.sqrt(a * a + rho * rho) - 1.0))


# ---------------------------------------------------------------------------------------
# Data-parallel semantics of Algorithm 2 (W workers emulated on one host)
# ---------------------------------------------------------------------------------------
# Worker w holds its own X^w, M^w, Q^w and prev_norm^w and computes its own gradient.  Each
# step: B^w = M^w + G^w and RMMC^w_l per layer (local); AllReduce_max of RMMC over workers (and
# over layers for the global flag); on a sync, P = AllReduce_DP(B^w Q^w), Orthogonalize(P),
# R = AllReduce_DP(B^w^T P), then each worker applies the same P, R, Q_t to its own M^w, X^w;
# otherwise each worker takes its local step.  AllReduce_DP is read as the mean over workers
# (the data-parallel average of Dion's reference implementation); with one worker it is the
# identity and this is curvadion_step.

@dataclass
class DPStepOutput:
    workers: List[List[LayerState]]
    prev_norm: List[np.ndarray]
    rmmc: List[np.ndarray]          # per worker, per layer (local)
    rmmc_max: np.ndarray            # per layer, max over workers (the AllReduce_max)
    flags: np.ndarray
    global_flag: bool
    active: np.ndarray


def curvadion_step_dp(workers: Sequence[Sequence[LayerState]], grads: Sequence[Sequence[np.ndarray]],
                      prev_norm: Sequence[Sequence[float]], hp: HParams, step: int) -> DPStepOutput:
    """One step of Algorithm 2 over W data-parallel workers (lists indexed [worker][layer])."""
    W = len(workers)
    L = len(workers[0]) if W else 0
    Bs = [[form_buffer(as_f64(workers[w][l].M), as_f64(grads[w][l])) for l in range(L)] for w in range(W)]
    nb = [np.array([frobenius_norm(Bs[w][l]) for l in range(L)]) for w in range(W)]
    rm = [np.array([rmmc_alg2(nb[w][l], float(prev_norm[w][l]), hp.eps_rmmc) for l in range(L)])
          for w in range(W)]
    rmax = np.array([max((rm[w][l] if math.isfinite(rm[w][l]) else math.inf) for w in range(W))
                     for l in range(L)])
    flags, gflag, active = gate(rmax, [workers[0][l].tau for l in range(L)], hp.tau_global, hp.gate_mode,
                                step, hp.period)
    out = [[None] * L for _ in range(W)]
    for l in range(L):
        if active[l]:
            P = sum(power_iter(Bs[w][l], as_f64(workers[w][l].Q)) for w in range(W)) / W
            P = orthogonalize(P)
            R = sum(Bs[w][l].T @ P for w in range(W)) / W
            Q_new = column_normalize(R, hp.eps_col)
            for w in range(W):
                st = workers[w][l]
                m, n = Bs[w][l].shape
                M_new = Bs[w][l] - (1.0 - hp.mu) * (P @ R.T)
                X_new = decay_parameters(as_f64(st.X), hp.eta, hp.weight_decay) - hp.eta * math.sqrt(m / n) * (P @ Q_new.T)
                out[w][l] = LayerState(X=X_new, M=M_new, Q=Q_new.copy(), tau=st.tau)
        else:
            for w in range(W):
                st = workers[w][l]
                M_new, X_new = local_update(Bs[w][l], as_f64(grads[w][l]), as_f64(st.X), hp.eta_local, hp.weight_decay)
                out[w][l] = LayerState(X=X_new, M=M_new, Q=as_f64(st.Q), tau=st.tau)
    return DPStepOutput(workers=out, prev_norm=[x.copy() for x in nb], rmmc=rm, rmmc_max=rmax,
                        flags=np.array(flags, dtype=bool), global_flag=bool(gflag), active=np.array(active, dtype=bool))
