"""Failure detection on the GPU without a fault: a bounded wait is made to run out.

Every wait between the roles of a tensor-core kernel (a TMA load landing, an MMA finishing, an
accumulator being drained) gives up after a limit, sets DION_ERR_TIMEOUT and lets the kernel
drain what it already issued and return, so the context stays usable.  The test shortens that
limit for the update kernel's hand-off waits to a few nanoseconds, so its first wait that does
not succeed at once gives up: nothing is broken, the wait simply runs out.  The host then reads
the status, restores the limit, and the next step matches the oracle from the device state.
"""
import pytest
import torch

import workloads as wl
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu

TOL_BF16 = 2e-2


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2512_13728_gb300 import build

    build.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"


def test_update_wait_runs_out_then_next_step_passes():
    import paper_2512_13728_gb300 as cd

    w = wl.scaled(wl.WORKLOADS["gpt160m_block_r192"], "timeout", [(512, 384), (384, 512), (200, 136)], rank=32,
                  steps=3)
    st = gu.make_state(w)
    plan = cd.Plan(st.X, st.M, st.Q, st.G, st.taus, cd.DION_PREC_BF16)
    hpo = gu.oracle_hp()
    try:
        # step 1 with the default limit
        gu.write_gradients(st, 1)
        plan.step(cd.hparams(step=1))
        torch.cuda.synchronize()
        assert plan.device_status() == 0
        # step 2: the update kernel's hand-off waits give up after 1 ns
        cd.native.dion_plan_set_wait_limit(plan.handle, 1)
        gu.write_gradients(st, 2)
        plan.step(cd.hparams(step=2))
        torch.cuda.synchronize()  # the kernel returned: the context is still usable
        assert plan.device_status() == cd.native.DION_ERR_TIMEOUT
        assert plan.device_status() == 0  # cleared by the read
        # step 3 with the default limit restored: parity with the oracle from the device state
        cd.native.dion_plan_set_wait_limit(plan.handle, 0)
        gu.write_gradients(st, 3)
        layers, grads, prev = gu.snapshot(st, plan)
        plan.step(cd.hparams(step=3))
        torch.cuda.synchronize()
        assert plan.device_status() == 0
        c = gu.compare_step(st, plan, layers, grads, prev, hpo, 3)
        assert max(c.err_M, c.err_X, c.err_Q) <= TOL_BF16, c
        assert c.flags_equal and c.gflag_equal
    finally:
        plan.close()

