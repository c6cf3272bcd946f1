"""Pins of the fp64 oracle against results fixed outside it (CPU only).

Each test checks the oracle against something it does not compute itself: LAPACK's QR,
brute force with scalar Python loops on tiny matrices, closed forms that follow from the
algorithms of the paper, and algebraic identities of the Dion update.  The mutation tests
at the end plant plausible mistakes in the oracle and require that some pin catches each.
"""
import math
import os

import numpy as np
import pytest

import oracle.curvadion as oc

RNG = np.random.default_rng(1234)
HERE = os.path.dirname(os.path.abspath(__file__))


def rel(a, b):
    return float(np.linalg.norm(np.asarray(a) - np.asarray(b)) / max(np.linalg.norm(b), 1e-300))


# ----------------------------------------------------------------- QR (Orthogonalize) ---

def lapack_qr_pos(A):
    q, r = np.linalg.qr(A, mode="reduced")
    d = np.where(np.diag(r) < 0, -1.0, 1.0)
    return q * d, r * d[:, None]


@pytest.mark.parametrize("m,r", [(4, 3), (7, 7), (64, 16), (300, 48), (129, 128), (33, 1)])
def test_householder_matches_lapack(m, r):
    A = RNG.standard_normal((m, r)) * RNG.uniform(0.1, 10.0, size=r)
    q, rr = oc.householder_qr(A)
    ql, rl = lapack_qr_pos(A)
    assert rel(q, ql) < 1e-11
    assert rel(rr, rl) < 1e-11


@pytest.mark.parametrize("m,r", [(10, 4), (200, 64), (64, 64)])
def test_householder_factorization_properties(m, r):
    A = RNG.standard_normal((m, r))
    q, rr = oc.householder_qr(A)
    assert np.allclose(q.T @ q, np.eye(r), atol=1e-12)  # orthonormal columns
    assert np.allclose(q @ rr, A, atol=1e-12)  # reconstructs the input
    assert np.allclose(rr, np.triu(rr))  # triangular factor
    assert np.all(np.diag(rr) > 0)  # positive diagonal


def test_householder_ill_conditioned_stays_orthonormal():
    u, _ = np.linalg.qr(RNG.standard_normal((120, 20)))
    v, _ = np.linalg.qr(RNG.standard_normal((20, 20)))
    A = (u * np.logspace(0, -9, 20)) @ v.T  # condition number 1e9
    q, rr = oc.householder_qr(A)
    assert np.abs(q.T @ q - np.eye(20)).max() < 1e-12
    assert rel(q @ rr, A) < 1e-13


# ----------------------------------------------------- brute force with scalar loops ---

def bf_matmul(A, B):
    n, k = len(A), len(A[0])
    m = len(B[0])
    return [[sum(A[i][p] * B[p][j] for p in range(k)) for j in range(m)] for i in range(n)]


def bf_T(A):
    return [list(col) for col in zip(*A)]


def bf_gram_schmidt(P):
    """Modified Gram-Schmidt on the columns of P (positive diagonal by construction)."""
    m, r = len(P), len(P[0])
    cols = [[P[i][j] for i in range(m)] for j in range(r)]
    out = []
    for j in range(r):
        v = cols[j][:]
        for q in out:
            d = sum(q[i] * v[i] for i in range(m))
            v = [v[i] - d * q[i] for i in range(m)]
        nv = math.sqrt(sum(x * x for x in v))
        out.append([x / nv for x in v])
    return [[out[j][i] for j in range(r)] for i in range(m)]


def bf_dion(B, Qp, X, mu, eta, eps_col):
    m, n = len(B), len(B[0])
    P = bf_gram_schmidt(bf_matmul(B, Qp))
    R = bf_matmul(bf_T(B), P)
    PRt = bf_matmul(P, bf_T(R))
    r = len(P[0])
    cn = [math.sqrt(sum(R[i][j] ** 2 for i in range(n))) for j in range(r)]
    Qn = [[R[i][j] / (cn[j] + eps_col) for j in range(r)] for i in range(n)]
    PQt = bf_matmul(P, bf_T(Qn))
    s = math.sqrt(m / n)
    Mn = [[B[i][j] - (1 - mu) * PRt[i][j] for j in range(n)] for i in range(m)]
    Xn = [[X[i][j] - eta * s * PQt[i][j] for j in range(n)] for i in range(m)]
    return np.array(Mn), np.array(Qn), np.array(Xn)


@pytest.mark.parametrize("m,n", [(4, 3), (3, 4)])
@pytest.mark.parametrize("r", [1, 2, 3])
def test_bruteforce_small_dion_update(m, n, r):
    B = RNG.standard_normal((m, n))
    Qp = RNG.standard_normal((n, r))
    X = RNG.standard_normal((m, n))
    mu, eta, eps = 0.9, 0.05, 1e-3
    res = oc.dion_sync_update(B, Qp, X, mu, eta, eps)
    Mb, Qb, Xb = bf_dion(B.tolist(), Qp.tolist(), X.tolist(), mu, eta, eps)
    assert rel(res.M, Mb) < 1e-12
    assert rel(res.Q, Qb) < 1e-12
    assert rel(res.X, Xb) < 1e-12


def test_bruteforce_step_rmmc_and_flags():
    """A 2-layer Algorithm 2 step checked against scalar loops for norm, RMMC and the gate."""
    shapes = [(4, 3), (3, 5)]
    layers = [oc.LayerState(X=RNG.standard_normal(s), M=RNG.standard_normal(s), Q=RNG.standard_normal((s[1], 2)),
                            tau=0.3) for s in shapes]
    grads = [RNG.standard_normal(s) for s in shapes]
    prev = [2.5, 7.0]
    hp = oc.HParams(gate_mode=oc.GATE_PER_LAYER, eps_rmmc=1e-3)
    out = oc.curvadion_step(layers, grads, prev, hp, step=3)
    for i, (st, G) in enumerate(zip(layers, grads)):
        m, n = shapes[i]
        nb = math.sqrt(sum((st.M[a][b] + G[a][b]) ** 2 for a in range(m) for b in range(n)))
        want = abs(nb - prev[i]) / (prev[i] + 1e-3)
        assert out.rmmc[i] == pytest.approx(want, rel=1e-13)
        assert out.prev_norm[i] == pytest.approx(nb, rel=1e-13)
        assert bool(out.flags[i]) == (want > 0.3)
        if not out.active[i]:  # local branch: M = B, X = X - eta_local G
            assert np.allclose(out.layers[i].M, st.M + G, atol=0, rtol=0)
            assert np.allclose(out.layers[i].X, st.X - hp.eta_local * G, rtol=1e-15)


# ------------------------------------------------------------ identities of the update ---

@pytest.mark.parametrize("m,n,r", [(40, 30, 5), (30, 40, 7), (64, 64, 16)])
def test_error_feedback_identity(m, n, r):
    """B = M_t + (1 - mu) P R^T and, since R^T = P^T B, P^T M_t = mu P^T B."""
    B = RNG.standard_normal((m, n))
    Qp = RNG.standard_normal((n, r))
    mu = 0.95
    res = oc.dion_sync_update(B, Qp, np.zeros((m, n)), mu, 0.01, 1e-8)
    assert rel(res.M + (1 - mu) * res.P @ res.R.T, B) < 1e-13
    assert rel(res.P.T @ res.M, mu * (res.P.T @ B)) < 1e-12
    assert np.allclose(res.P.T @ res.P, np.eye(r), atol=1e-12)


@pytest.mark.parametrize("m,n", [(12, 8), (8, 12), (10, 10)])
def test_full_rank_recovers_buffer(m, n):
    """r = min(m, n): the projection P P^T B (or B Q Q^T) is B itself, so M_t = mu B."""
    r = min(m, n)
    B = RNG.standard_normal((m, n))
    res = oc.dion_sync_update(B, RNG.standard_normal((n, r)), np.zeros((m, n)), 0.9, 0.01, 1e-8)
    assert rel(res.P @ res.R.T, B) < 1e-12
    assert rel(res.M, 0.9 * B) < 1e-12


def test_unit_column_norms():
    B = RNG.standard_normal((50, 40))
    res = oc.dion_sync_update(B, RNG.standard_normal((40, 6)), np.zeros((50, 40)), 0.95, 0.01, 1e-8)
    cn = np.linalg.norm(res.R, axis=0)
    assert np.allclose(np.linalg.norm(res.Q, axis=0), cn / (cn + 1e-8), rtol=1e-14)


@pytest.mark.parametrize("m,n", [(6, 11), (11, 6)])
def test_rank_one_closed_form(m, n):
    """B = s u v^T, r = 1, v^T q > 0:  P = u, R = s v, Q = v s/(s+eps), M = mu B,
    X_t = X - eta sqrt(m/n) u v^T s/(s + eps).  m != n pins the sqrt(m/n) factor."""
    u = RNG.standard_normal(m); u /= np.linalg.norm(u)
    v = RNG.standard_normal(n); v /= np.linalg.norm(v)
    s, mu, eta, eps = 3.0, 0.95, 0.02, 1e-2
    q = v + 0.1 * RNG.standard_normal(n)
    X = RNG.standard_normal((m, n))
    res = oc.dion_sync_update(s * np.outer(u, v), q[:, None], X, mu, eta, eps)
    assert rel(res.P[:, 0], u) < 1e-13
    assert rel(res.R[:, 0], s * v) < 1e-13
    assert rel(res.Q[:, 0], v * s / (s + eps)) < 1e-13
    assert rel(res.M, mu * s * np.outer(u, v)) < 1e-13
    assert rel(res.X, X - eta * math.sqrt(m / n) * (s / (s + eps)) * np.outer(u, v)) < 1e-13


def test_rank_k_gradients_follow_momentum_recurrence():
    """G_t = c_t U V^T (rank k) and r = k: Dion is exact, so B_{t+1} = mu B_t + G_{t+1}."""
    m, n, k, mu = 30, 20, 3, 0.9
    U = RNG.standard_normal((m, k)); V = RNG.standard_normal((n, k))
    cs = [1.0, -0.5, 2.0, 0.7, 1.3]
    layer = oc.LayerState(X=np.zeros((m, n)), M=np.zeros((m, n)), Q=RNG.standard_normal((n, k)))
    hp = oc.HParams(mu=mu, gate_mode=oc.GATE_ALWAYS)
    _, outs = oc.run_trajectory([layer], lambda i, t: cs[t - 1] * U @ V.T, len(cs), hp)
    b = 0.0
    for t, o in enumerate(outs, start=1):
        b = mu * b + cs[t - 1]  # scalar recurrence of the coefficient of U V^T
        assert o.norm_b[0] == pytest.approx(abs(b) * np.linalg.norm(U @ V.T), rel=1e-11)
        assert rel(o.layers[0].M, mu * b * U @ V.T) < 1e-11


# --------------------------------------------------------------- RMMC closed forms ---

def load_golden():
    rows = []
    with open(os.path.join(HERE, "golden", "rmmc_closed_form_mu095.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            t, a, b = line.split()
            rows.append((int(t), float(a), float(b)))
    return rows


def test_rmmc_constant_gradient_dion_full_rank_matches_golden():
    m, n = 9, 6
    G = RNG.standard_normal((m, n))
    layer = oc.LayerState(X=np.zeros((m, n)), M=np.zeros((m, n)), Q=RNG.standard_normal((n, n)), tau=0.5)
    hp = oc.HParams(mu=0.95, eps_rmmc=1e-30, gate_mode=oc.GATE_ALWAYS)
    _, outs = oc.run_trajectory([layer], lambda i, t: G, 12, hp)
    for t, want, _ in load_golden():
        assert outs[t - 1].rmmc[0] == pytest.approx(want, rel=1e-10)
        assert bool(outs[t - 1].flags[0]) == (want > 0.5)
    # first step: prev_norm = 0, so RMMC_1 = ||G|| / eps and the layer synchronizes
    assert outs[0].rmmc[0] == pytest.approx(np.linalg.norm(G) / 1e-30, rel=1e-12)


def test_rmmc_constant_gradient_local_only_matches_golden():
    m, n = 5, 7
    G = RNG.standard_normal((m, n))
    X0 = RNG.standard_normal((m, n))
    layer = oc.LayerState(X=X0, M=np.zeros((m, n)), Q=RNG.standard_normal((n, 2)), tau=math.inf)
    hp = oc.HParams(eps_rmmc=1e-30, eta_local=0.03, gate_mode=oc.GATE_PER_LAYER)
    last, outs = oc.run_trajectory([layer], lambda i, t: G, 12, hp)
    for t, _, want in load_golden():
        assert outs[t - 1].rmmc[0] == pytest.approx(want, rel=1e-10)
    assert rel(last[0].M, 12 * G) < 1e-14
    assert rel(last[0].X, X0 - 12 * 0.03 * G) < 1e-13


def test_eq1_equals_alg2_under_full_rank():
    """Full-rank Dion: M_t = mu B_t, so Equation 1 on M equals Algorithm 2 on B for t >= 2."""
    m, n = 8, 8
    layer = oc.LayerState(X=np.zeros((m, n)), M=np.zeros((m, n)), Q=RNG.standard_normal((n, n)))
    hp = oc.HParams(mu=0.9, eps_rmmc=1e-30)
    _, outs = oc.run_trajectory([layer], lambda i, t: RNG.standard_normal((m, n)), 6, hp)
    for t in range(2, 6):
        # Eq.1 at step t compares ||M_t|| with ||M_{t-1}||; Alg.2 at step t+1 compares ||B_{t+1}||...
        # both reduce to the same ratio of consecutive buffer norms:
        eq1 = outs[t - 1].rmmc_eq1[0]
        alg2 = outs[t - 1].rmmc[0]
        assert eq1 == pytest.approx(alg2, rel=1e-10)


# ------------------------------------------------------------------------- the gate ---

def test_gate_strict_threshold_and_modes():
    rm = [0.5, 0.2, 0.7]
    taus = [0.5, 0.1, 0.9]
    flags, g, act = oc.gate(rm, taus, 0.6, oc.GATE_PER_LAYER, step=1, period=1)
    assert flags == [False, True, False]  # 0.5 > 0.5 is false: strict compare
    assert act == flags
    assert g is True  # max 0.7 > 0.6
    _, g2, act2 = oc.gate(rm, taus, 0.7, oc.GATE_GLOBAL, 1, 1)
    assert g2 is False and act2 == [False] * 3
    _, _, act3 = oc.gate(rm, taus, 0.7, oc.GATE_ALWAYS, 1, 1)
    assert act3 == [True] * 3
    for step in range(1, 13):
        _, _, a = oc.gate(rm, taus, 0.7, oc.GATE_SCHEDULED, step, 4)
        assert a == [step % 4 == 0] * 3


def test_gate_nonfinite_is_above():
    flags, g, act = oc.gate([float("nan"), 0.0], [0.5, 0.5], 0.5, oc.GATE_GLOBAL, 1, 1)
    assert flags == [True, False] and g is True and act == [True, True]


# -------------------------------------------------- mutation tests: pins have teeth ---

def _pins_fail(monkeypatch, name, fake, pins):
    monkeypatch.setattr(oc, name, fake)
    failed = 0
    for pin in pins:
        try:
            pin()
        except AssertionError:
            failed += 1
    monkeypatch.undo()
    return failed


def test_mutation_wrong_decay_is_caught(monkeypatch):
    real = oc.dion_sync_update

    def mutated(B, Qp, X, mu, eta, eps_col, weight_decay=0.0):  # (1 - mu) replaced by mu
        return real(B, Qp, X, 1.0 - mu, eta, eps_col, weight_decay)

    assert _pins_fail(monkeypatch, "dion_sync_update", mutated,
                      [lambda: test_full_rank_recovers_buffer(12, 8)]) == 1


def test_mutation_missing_sign_fix_is_caught(monkeypatch):
    def mutated(A):
        q, r = np.linalg.qr(A)
        return q, r

    assert _pins_fail(monkeypatch, "householder_qr", mutated,
                      [lambda: test_householder_factorization_properties(10, 4)]) == 1


def test_mutation_transposed_scale_is_caught(monkeypatch):
    def mutated(B, Qp, X, mu, eta, eps_col, weight_decay=0.0):  # sqrt(n/m) instead of sqrt(m/n)
        m, n = B.shape
        P = oc.orthogonalize(B @ Qp)
        R = B.T @ P
        Qn = oc.column_normalize(R, eps_col)
        return oc.SyncResult(M=B - (1 - mu) * P @ R.T, Q=Qn, X=X - eta * math.sqrt(n / m) * P @ Qn.T, P=P, R=R)

    assert _pins_fail(monkeypatch, "dion_sync_update", mutated,
                      [lambda: test_rank_one_closed_form(6, 11)]) == 1


def test_mutation_stale_q_in_update_is_caught(monkeypatch):
    def mutated(B, Qp, X, mu, eta, eps_col, weight_decay=0.0):  # parameter update with Q_{t-1} instead of Q_t
        m, n = B.shape
        P = oc.orthogonalize(B @ Qp)
        R = B.T @ P
        Qn = oc.column_normalize(R, eps_col)
        return oc.SyncResult(M=B - (1 - mu) * P @ R.T, Q=Qn, X=X - eta * math.sqrt(m / n) * P @ Qp.T, P=P, R=R)

    assert _pins_fail(monkeypatch, "dion_sync_update", mutated,
                      [lambda: test_bruteforce_small_dion_update(4, 3, 2)]) == 1


def test_mutation_rmmc_without_abs_is_caught(monkeypatch):
    def mutated(nb, prev, eps):
        return (nb - prev) / (prev + eps)

    # the local-only sequence grows (positive change); a decreasing sequence needs the abs:
    def pin_decreasing():
        m, n = 4, 4
        G = RNG.standard_normal((m, n))
        layer = oc.LayerState(X=np.zeros((m, n)), M=5 * G, Q=np.eye(n)[:, :2], tau=math.inf)
        hp = oc.HParams(eps_rmmc=1e-30, gate_mode=oc.GATE_PER_LAYER)
        o = oc.curvadion_step([layer], [-G], [np.linalg.norm(5 * G)], hp, 2)
        assert o.rmmc[0] == pytest.approx(0.2, rel=1e-12)  # ||4G|| vs ||5G||

    pin_decreasing()
    assert _pins_fail(monkeypatch, "rmmc_alg2", mutated, [pin_decreasing]) == 1


# ------------------------------------------- training-loop fidelity (Section 4 settings) ---

@pytest.mark.parametrize("m,n,r", [(6, 9, 3), (12, 5, 5)])
def test_weight_decay_is_decoupled(m, n, r):
    """Decoupled decay changes only X, and by exactly -lr * wd * X in both branches; M, Q, P, R
    are those of the undecayed step (the decay never enters the momentum)."""
    B = RNG.standard_normal((m, n))
    Qp = RNG.standard_normal((n, r))
    X = RNG.standard_normal((m, n))
    G = RNG.standard_normal((m, n))
    a = oc.dion_sync_update(B, Qp, X, 0.9, 0.05, 1e-8, 0.0)
    b = oc.dion_sync_update(B, Qp, X, 0.9, 0.05, 1e-8, 0.3)
    assert np.array_equal(a.M, b.M) and np.array_equal(a.Q, b.Q) and np.array_equal(a.P, b.P)
    assert np.allclose(b.X - a.X, -0.05 * 0.3 * X, rtol=0, atol=1e-14)
    M0, X0 = oc.local_update(B, G, X, 0.07, 0.0)
    M1, X1 = oc.local_update(B, G, X, 0.07, 0.3)
    assert np.array_equal(M0, M1)
    assert np.allclose(X1 - X0, -0.07 * 0.3 * X, rtol=0, atol=1e-14)


def test_weight_decay_local_steps_closed_form():
    """With zero gradients every local step only decays: X_t = (1 - eta_local wd)^t X_0 (scalar
    loop check), and M stays 0."""
    m, n = 3, 4
    X0 = RNG.standard_normal((m, n))
    layer = oc.LayerState(X=X0.copy(), M=np.zeros((m, n)), Q=np.eye(n)[:, :2], tau=math.inf)
    hp = oc.HParams(eta_local=0.1, weight_decay=0.5, gate_mode=oc.GATE_PER_LAYER)
    cur, prev = [layer], [0.0]
    for t in range(1, 6):
        o = oc.curvadion_step(cur, [np.zeros((m, n))], prev, hp, t)
        cur, prev = o.layers, o.prev_norm
    for i in range(m):
        for j in range(n):
            v = X0[i, j]
            for _ in range(5):
                v = v * (1.0 - 0.1 * 0.5)
            assert cur[0].X[i, j] == pytest.approx(v, rel=1e-14, abs=1e-300)
    assert not np.any(cur[0].M)


@pytest.mark.parametrize("T,wu,wd", [(3000, 0.01, 0.2), (3000, 0.01, 0.1), (100, 0.0, 0.5), (50, 0.1, 0.0)])
def test_lr_schedule_shape(T, wu, wd):
    """Section 4's schedule: linear rise to the base rate over round(wu T) steps, flat, linear fall
    to exactly 0 at the last step over round(wd T) steps; every piece is affine in the step."""
    base = 0.02
    lr = np.array([oc.lr_schedule(t, T, base, wu, wd) for t in range(1, T + 1)])
    W, D = int(math.floor(wu * T + 0.5)), int(math.floor(wd * T + 0.5))
    assert np.all(lr >= 0) and np.all(lr <= base)
    if D > 0:
        assert lr[-1] == 0.0
        assert lr[T - D - 1] == base  # last flat step
        fall = lr[T - D - 1:]
        assert np.allclose(np.diff(fall, 2), 0.0, atol=1e-15) and np.all(np.diff(fall) < 0)
    else:
        assert lr[-1] == base
    if W > 0:
        rise = np.concatenate([[0.0], lr[:W]])
        assert lr[W - 1] == base and np.allclose(np.diff(rise, 2), 0.0, atol=1e-15)
        assert lr[0] == pytest.approx(base / W)
    flat = lr[W:T - D]
    assert np.all(flat == base)
    # outside [1, T] the schedule clamps
    assert oc.lr_schedule(0, T, base, wu, wd) == lr[0] and oc.lr_schedule(T + 5, T, base, wu, wd) == lr[-1]


@pytest.mark.parametrize("m,n,f,r", [(768, 3072, 0.125, 96), (2048, 8192, 0.125, 256), (100, 100, 0.125, 13),
                                     (1, 5, 0.125, 1), (64, 64, 1.0, 64), (4096, 1024, 1 / 16, 64),
                                     (768, 768, 0.25, 192)])
def test_rank_for(m, n, f, r):
    assert oc.rank_for(m, n, f) == r


def test_mutation_decay_after_update_is_caught(monkeypatch):
    real = oc.dion_sync_update

    def mutated(B, Qp, X, mu, eta, eps_col, weight_decay=0.0):  # decays the updated X instead of X
        res = real(B, Qp, X, mu, eta, eps_col, 0.0)
        res.X = (1.0 - eta * weight_decay) * res.X
        return res

    assert _pins_fail(monkeypatch, "dion_sync_update", mutated,
                      [lambda: test_weight_decay_is_decoupled(6, 9, 3)]) == 1
