"""Data-parallel semantics of Algorithm 2 (W workers) in the oracle, CPU only.

Pins of ``curvadion_step_dp`` against results it does not compute itself: one worker is
``curvadion_step``; the sync branch depends on the workers' buffers only through their mean
(P and R are linear in B before Orthogonalize), so W workers with shared state equal one worker
fed the mean gradient; one worker's spike makes every worker sync (the AllReduce_max); local
steps let the workers drift apart with no exchange.  A 2-rank gloo run of the same step with
real collectives is in ``test_dp_gloo.py``.
"""
import numpy as np
import pytest

import oracle.curvadion as oc

RNG = np.random.default_rng(2024)
SHAPES = [(24, 16), (16, 40), (9, 9)]
RANKS = [4, 3, 9]


def states(seed, shared=None):
    g = np.random.default_rng(seed)
    out = []
    for (m, n), r in zip(SHAPES, RANKS):
        q = g.standard_normal((n, r))
        q /= np.linalg.norm(q, axis=0, keepdims=True)
        out.append(oc.LayerState(X=g.standard_normal((m, n)), M=0.1 * g.standard_normal((m, n)), Q=q, tau=0.5))
    if shared is not None:  # same X, M, Q as `shared`
        out = [oc.LayerState(X=s.X.copy(), M=s.M.copy(), Q=s.Q.copy(), tau=s.tau) for s in shared]
    return out


def grads(seed, scale=1.0):
    g = np.random.default_rng(seed)
    return [scale * g.standard_normal(s) for s in SHAPES]


@pytest.mark.parametrize("mode", [oc.GATE_ALWAYS, oc.GATE_GLOBAL, oc.GATE_PER_LAYER])
def test_one_worker_is_the_single_worker_step(mode):
    st, G = states(1), grads(2)
    prev = [0.3, 2.0, 1.0]
    hp = oc.HParams(gate_mode=mode, weight_decay=0.1)
    a = oc.curvadion_step(st, G, prev, hp, 3)
    b = oc.curvadion_step_dp([st], [G], [prev], hp, 3)
    assert np.array_equal(a.active, b.active) and np.array_equal(a.flags, b.flags) and a.global_flag == b.global_flag
    assert np.array_equal(a.rmmc, b.rmmc[0])
    for x, y in zip(a.layers, b.workers[0]):
        for f in ("X", "M", "Q"):
            assert np.allclose(getattr(x, f), getattr(y, f), rtol=0, atol=1e-13)


def test_sync_depends_on_the_mean_buffer():
    """W = 3 workers with the same X, M, Q and different gradients, all syncing: P, R and so Q_t
    and every worker's X_t are those of one worker fed the mean gradient, and the workers' mean
    M_t is that worker's M_t (Algorithm 2's AllReduce_DP lines are linear in B)."""
    base = states(5)
    ws = [states(0, shared=base) for _ in range(3)]
    Gs = [grads(10 + w) for w in range(3)]
    Gmean = [sum(Gs[w][l] for w in range(3)) / 3 for l in range(len(SHAPES))]
    hp = oc.HParams(gate_mode=oc.GATE_ALWAYS, weight_decay=0.05)
    dp = oc.curvadion_step_dp(ws, Gs, [[0.0] * 3] * 3, hp, 1)
    one = oc.curvadion_step(base, Gmean, [0.0] * 3, hp, 1)
    for l in range(len(SHAPES)):
        for w in range(3):
            assert np.allclose(dp.workers[w][l].X, one.layers[l].X, rtol=0, atol=1e-12)
            assert np.allclose(dp.workers[w][l].Q, one.layers[l].Q, rtol=0, atol=1e-12)
        Mmean = sum(dp.workers[w][l].M for w in range(3)) / 3
        assert np.allclose(Mmean, one.layers[l].M, rtol=0, atol=1e-12)


def test_one_workers_spike_syncs_everyone():
    """GATE_GLOBAL: worker 1's large gradient change lifts the AllReduce_max above tau for all."""
    base = states(7)
    ws = [states(0, shared=base) for _ in range(2)]
    prev = [[float(np.linalg.norm(s.M)) for s in base]] * 2  # as if the last buffers were M
    calm = [0.01 * g for g in grads(3)]
    Gs = [calm, [g.copy() for g in calm]]
    Gs[1][2] = 50.0 * grads(4)[2]
    hp = oc.HParams(gate_mode=oc.GATE_GLOBAL, tau_global=0.5)
    quiet = oc.curvadion_step_dp(ws, [calm, calm], prev, hp, 2)
    loud = oc.curvadion_step_dp(ws, Gs, prev, hp, 2)
    assert not quiet.global_flag and not quiet.active.any()
    assert loud.global_flag and loud.active.all()
    assert loud.rmmc_max[2] == max(loud.rmmc[0][2], loud.rmmc[1][2]) > 0.5
    assert loud.rmmc[0][2] < 0.5  # worker 0 alone would not have synced


def test_local_steps_diverge_without_exchange():
    base = states(9)
    ws = [states(0, shared=base) for _ in range(2)]
    Gs = [grads(20), grads(21)]
    hp = oc.HParams(gate_mode=oc.GATE_PER_LAYER, eta_local=0.07, weight_decay=0.1)
    for s in ws[0] + ws[1]:
        s.tau = np.inf
    dp = oc.curvadion_step_dp(ws, Gs, [[1e9] * 3] * 2, hp, 2)
    assert not dp.active.any()
    for w in range(2):
        solo = oc.curvadion_step(ws[w], Gs[w], [1e9] * 3, hp, 2)
        for l in range(len(SHAPES)):
            assert np.array_equal(dp.workers[w][l].X, solo.layers[l].X)
            assert np.array_equal(dp.workers[w][l].M, solo.layers[l].M)
    assert not np.allclose(dp.workers[0][0].X, dp.workers[1][0].X)
