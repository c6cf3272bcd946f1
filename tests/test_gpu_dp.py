"""Data-parallel steps through the C ABI's phases (Algorithm 2 with W workers).

Each worker is one plan.  Between the phases the test performs Algorithm 2's reductions itself,
on the device with torch: the elementwise maximum of RMMC after DION_PHASE_NORMS, the mean of the
P range after DION_PHASE_POWER and of the R range after DION_PHASE_ORTHO (what NCCL would do
across GPUs).  No kernel waits for another worker: the host orders the phases on one stream.
The results are compared step by step with the oracle's W-worker step from the device state.
"""
import math

import numpy as np
import pytest
import torch

import oracle.curvadion as oc
import workloads as wl
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu

TOL = {"fp32": 1e-4, "bf16": 2e-2, "bf16x3": 1e-4}
PRECS = {"fp32": 0, "bf16": 1, "bf16x3": 2}
SHAPES = [(200, 136), (136, 200), (264, 264), (67, 33)]


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2512_13728_gb300 import build

    build.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"


def worker_workload(w, g_dtype):
    """Worker w's gradients: the same shapes and statistics, its own seed; worker 1's gradients
    spike (x8) at step 4, so that one worker's RMMC makes every worker synchronize."""
    base = wl.scaled(wl.WORKLOADS["gpt160m_block_r192"], f"dp{w}", SHAPES, rank=24, steps=6, g_dtype=g_dtype)
    return wl.scaled(base, f"dp{w}", SHAPES, seed=100 + w)


def gradient(w, l, t, dev, g_dtype):
    g = wl.gradient(worker_workload(w, g_dtype), l, t, dev)
    return g * 8 if (w == 1 and t == 4) else g


def run_workers(W, prec, gate_mode, taus, g_dtype="bf16", steps=6):
    import paper_2512_13728_gb300 as cd

    base = worker_workload(0, g_dtype)
    states = [gu.make_state(base, taus=taus) for _ in range(W)]  # identical X_0, M_0, Q_0
    plans = [cd.Plan(s.X, s.M, s.Q, s.G, s.taus, PRECS[prec]) for s in states]
    hp = cd.hparams(gate_mode=gate_mode, tau_global=0.5)
    hpo = gu.oracle_hp(gate_mode=gate_mode, tau_global=0.5)
    L = len(SHAPES)
    worst = dict(M=0.0, X=0.0, Q=0.0)
    synced = []
    try:
        for t in range(1, steps + 1):
            for w, s in enumerate(states):
                for l in range(L):
                    s.G[l].copy_(gradient(w, l, t, s.G[l].device, g_dtype))
            snap = [gu.snapshot(s, p) for s, p in zip(states, plans)]
            hp.step = t
            for p in plans:
                p.step_phase(cd.DION_PHASE_NORMS, hp)
            rmax = torch.stack([torch.nan_to_num(p.rmmc[:L], nan=math.inf) for p in plans]).amax(0)
            for p in plans:
                p.rmmc[:L].copy_(rmax)
            for p in plans:
                p.step_phase(cd.DION_PHASE_POWER, hp)
            for phase in (cd.DION_PHASE_POWER, cd.DION_PHASE_ORTHO):
                if phase == cd.DION_PHASE_ORTHO:
                    for p in plans:
                        p.step_phase(cd.DION_PHASE_ORTHO, hp)
                bufs = [p.exchange(phase) for p in plans]
                mean = torch.stack(bufs).mean(0)
                for b in bufs:
                    b.copy_(mean)
            for p in plans:
                p.step_phase(cd.DION_PHASE_UPDATE, hp)
            torch.cuda.synchronize()
            for p in plans:
                assert p.device_status() == 0
            want = oc.curvadion_step_dp([sn[0] for sn in snap], [sn[1] for sn in snap], [sn[2] for sn in snap],
                                        hpo, t)
            for w, (s, p) in enumerate(zip(states, plans)):
                assert np.array_equal(p.flags[:L].cpu().numpy().astype(bool), want.flags), (t, w)
                assert bool(p.global_flag[0].item()) == want.global_flag, (t, w)
                # norms from fp32 partial sums folded into fp64: 1e-5 relative (absolute below 1 for RMMC)
                got_pn = p.prev_norm[:L].double().cpu().numpy()
                assert np.allclose(got_pn, want.prev_norm[w], rtol=1e-5, atol=0), (t, w)
                rm = p.rmmc[:L].double().cpu().numpy()
                fin = np.isfinite(want.rmmc_max)
                err = np.abs(rm[fin] - want.rmmc_max[fin]) / np.maximum(np.abs(want.rmmc_max[fin]), 1.0)
                assert np.all(err <= 1e-5), (t, w, err)
                for l in range(L):
                    o = want.workers[w][l]
                    worst["M"] = max(worst["M"], gu.rel_fro(oc.as_f64(s.M[l]), o.M))
                    worst["X"] = max(worst["X"], gu.rel_fro(oc.as_f64(s.X[l]), o.X))
                    worst["Q"] = max(worst["Q"], gu.rel_fro(oc.as_f64(s.Q[l]), o.Q))
            assert max(worst.values()) <= TOL[prec], (t, worst)
            synced.append(int(want.active.sum()))
    finally:
        for p in plans:
            p.close()
    return worst, synced


@pytest.mark.parametrize("prec", ["fp32", "bf16", "bf16x3"])
def test_one_worker_phases_match_oracle(prec):
    """W = 1: the reductions are the identity and the phased step is Algorithm 2's step."""
    worst, synced = run_workers(1, prec, oc.GATE_PER_LAYER, [0.5, 0.3, 0.9, 0.5])
    print(prec, "one worker", worst, synced)


@pytest.mark.parametrize("prec,g_dtype", [("fp32", "fp32"), ("bf16", "bf16"), ("bf16", "fp32"), ("bf16x3", "bf16")])
@pytest.mark.parametrize("mode", ["global", "per_layer"])
def test_two_workers_emulated_on_one_gpu(prec, g_dtype, mode):
    """W = 2 workers with their own gradients (worker 1 spikes at step 4): flags from the maximum
    of the workers' RMMC, P and R averaged, per-worker error feedback; both workers against
    the oracle's two-worker step, with both branches taken."""
    gm = oc.GATE_GLOBAL if mode == "global" else oc.GATE_PER_LAYER
    worst, synced = run_workers(2, prec, gm, [0.5, 0.3, 0.9, 0.5], g_dtype=g_dtype)
    print(prec, g_dtype, mode, "two workers", worst, synced)
    assert synced[0] == len(SHAPES) and min(synced) < len(SHAPES)


def test_phase_order_is_enforced():
    import paper_2512_13728_gb300 as cd

    st = gu.make_state(worker_workload(0, "bf16"))
    gu.write_gradients(st, 1)
    plan = cd.Plan(st.X, st.M, st.Q, st.G, st.taus, cd.DION_PREC_BF16)
    try:
        hp = cd.hparams(step=1)
        with pytest.raises(cd.DionError):
            plan.step_phase(cd.DION_PHASE_POWER, hp)  # NORMS must come first
        plan.step_phase(cd.DION_PHASE_NORMS, hp)
        with pytest.raises(cd.DionError):
            plan.step(hp)  # a phased step is unfinished
        for ph in (cd.DION_PHASE_POWER, cd.DION_PHASE_ORTHO, cd.DION_PHASE_UPDATE):
            plan.step_phase(ph, hp)
        plan.step(cd.hparams(step=2))
        torch.cuda.synchronize()
        assert plan.device_status() == 0
        assert plan.exchange(cd.DION_PHASE_POWER).numel() >= sum(m * 24 for m, _ in SHAPES)
    finally:
        plan.close()
