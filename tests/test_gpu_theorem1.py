"""Theorem 1 validation workload on the GPU (the library's CurvaDion step, closed loop).

Four vector parameters (1 x n, n = 1, 64, 512, 2048; rank 1) descend F(x) = x^T H x / 2; each
step's gradient H x_t is formed from the device parameters and handed to dion_step.  Every
step is checked against the oracle's step from the same device state (X, M, Q to the mode's
tolerance, RMMC to 1e-5), and the device's RMMC is checked against Theorem 1's decomposition:
the exact momentum-norm ratio |sqrt((1 - B_t - eta kappa)^2 + rho^2) - 1| (to the mode's
accuracy) and |eta kappa + B_t| within the perpendicular-gradient term.
"""
import pytest
import torch

import oracle.curvadion as oc
import workloads as wl
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu

TOL_FP32, TOL_BF16, RMMC_RTOL = 1e-4, 2e-2, 1e-5


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2512_13728_gb300 import build

    build.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
def test_quadratic_closed_loop(prec):
    import paper_2512_13728_gb300 as cd

    p = cd.DION_PREC_FP32 if prec == "fp32" else cd.DION_PREC_BF16
    tol = TOL_FP32 if prec == "fp32" else TOL_BF16
    allow = 1e-3 if prec == "fp32" else 5e-2  # accuracy of the device RMMC against the exact ratio
    w = wl.Workload("quadratic", wl.QUADRATIC_SHAPES, 1, 30, "fp32", 0.0, seed=21)
    eta, mu, eps_col = 0.02, 0.95, 1e-8
    st = gu.make_state(w)
    H = []
    for l, (m, n) in enumerate(w.shapes):
        H.append(wl.quadratic_hessian(n, 300 + l, device="cuda"))
        st.X[l].copy_(wl.quadratic_start(n, 400 + l, device="cuda"))
    plan = cd.Plan(st.X, st.M, st.Q, st.G, st.taus, p)
    hpo = gu.oracle_hp(mu=mu, eta=eta, eps_col=eps_col)
    H64 = [h.double().cpu().numpy() for h in H]
    prev_snap = None
    worst_id, rows = 0.0, []
    try:
        for t in range(1, w.steps + 1):
            for l in range(w.num_layers):
                st.G[l].copy_(wl.quadratic_gradient(H[l], st.X[l]))
            layers, grads, prev = gu.snapshot(st, plan)
            plan.step(cd.hparams(step=t, mu=mu, eta=eta, eps_col=eps_col))
            torch.cuda.synchronize()
            assert plan.device_status() == 0
            c = gu.compare_step(st, plan, layers, grads, prev, hpo, t)
            assert c.err_M <= tol and c.err_X <= tol and c.err_Q <= tol, (t, c.err_M, c.err_X, c.err_Q)
            assert c.err_rmmc <= RMMC_RTOL, (t, c.err_rmmc)
            rm = plan.rmmc[: w.num_layers].double().cpu().numpy()
            if prev_snap is not None:
                pl, pg = prev_snap
                for l, (m, n) in enumerate(w.shapes):
                    b_prev = pl[l].M + pg[l]
                    terms = oc.theorem1_terms(H64[l], pl[l].X, b_prev, gu.f32(mu),
                                              oc.rank1_step_size(gu.f32(eta), n, b_prev, gu.f32(eps_col)))
                    a = 1.0 - terms.bias - terms.eta_eff * terms.kappa
                    assert a > 0
                    scale = max(terms.exact, 1e-3)
                    worst_id = max(worst_id, abs(rm[l] - terms.exact) / scale)
                    bound = terms.rho ** 2 / (2 * a)
                    # Theorem 1's first-order form, within the perpendicular-gradient term
                    assert abs(rm[l] - terms.prediction) <= bound + allow * scale + 1e-6, (t, n)
                    rows.append((t, n, rm[l], terms.prediction, terms.exact, bound))
            prev_snap = (layers, grads)
    finally:
        plan.close()
    # the device RMMC follows the exact decomposition (fp32: the step's rounding; bf16: the
    # bf16 operands of the parameter step move x_t by ~1e-3 relative)
    assert worst_id <= allow, worst_id
    for t, n, got, pred, exact, bound in rows[-4:]:
        print(f"t={t} n={n} RMMC={got:.6f} |eta kappa + B|={pred:.6f} exact={exact:.6f} rho^2/2a={bound:.2e}")
