"""Workspace guards and the DION_DEBUG_CHECKS build on the GPU.

Every region of a plan's workspace is followed by guard words; a kernel that wrote past its
region would change them.  The same sequence of steps (ragged shapes with NaN-padded rows, every
precision, a gated mode, a phased data-parallel step, host gradients) runs with the default
library and, in a child process, with libcurvadion_debug.so, which also checks the guards at the
end of every step and the tiles every kernel decodes.  Both leave every guard intact, the debug
build reports no error, and both produce the same bits.
"""
import os
import subprocess
import sys

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
pytestmark = pytest.mark.gpu


def run_sequence(out_path):
    """Runs the steps with whichever library native.py loads; saves the final state."""
    sys.path.insert(0, ROOT)
    import paper_2512_13728_gb300 as cd
    import workloads as wl
    from tests import gpu_util as gu

    w = wl.scaled(wl.WORKLOADS["gpt160m_block_r192"], "guards", [(200, 136), (136, 200), (264, 264), (67, 33),
                                                                 (1, 5), (5, 1)], rank=24, steps=3)
    results, damaged = [], []
    for prec, g_dtype, gate in [(0, "fp32", cd.DION_GATE_ALWAYS), (1, "bf16", cd.DION_GATE_ALWAYS),
                                (1, "bf16", cd.DION_GATE_PER_LAYER), (1, "fp32", cd.DION_GATE_ALWAYS),
                                (2, "bf16", cd.DION_GATE_GLOBAL)]:
        ws = wl.scaled(w, "guards", w.shapes, g_dtype=g_dtype)
        st = gu.make_state(ws, pad=1, taus=[0.5, 0.3, 1e6, 1e-6, 0.5, 0.5])
        plan = cd.Plan(st.X, st.M, st.Q, st.G, st.taus, prec)
        for t in range(1, ws.steps + 1):
            gu.write_gradients(st, t)
            plan.step(cd.hparams(step=t, gate_mode=gate))
        gu.write_gradients(st, ws.steps + 1)  # one phased step
        hp = cd.hparams(step=ws.steps + 1, gate_mode=gate)
        for ph in (cd.DION_PHASE_NORMS, cd.DION_PHASE_POWER, cd.DION_PHASE_ORTHO, cd.DION_PHASE_UPDATE):
            plan.step_phase(ph, hp)
        plan.enable_host_gradients()  # and one step with host gradients
        plan.step_host(cd.hparams(step=ws.steps + 2, gate_mode=gate), [g.cpu() for g in st.G])
        torch.cuda.synchronize()
        assert plan.device_status() == 0, (prec, g_dtype, gate)
        damaged.append(plan.check_guards())
        results += [x.cpu() for x in st.X + st.M + st.Q]
        plan.close()
    torch.save({"results": results, "damaged": damaged, "debug": cd.native.dion_debug_checks()}, out_path)


@pytest.fixture(scope="module")
def libs():
    from paper_2512_13728_gb300 import build

    return build.build(), build.build(debug=True)


def test_guards_intact_default_and_debug_builds(libs, tmp_path):
    _, debug_lib = libs
    a, b = tmp_path / "default.pt", tmp_path / "debug.pt"
    run_sequence(str(a))
    env = dict(os.environ, CURVADION_LIB=debug_lib)
    code = "import sys; sys.path.insert(0, %r); from tests.test_gpu_guards import run_sequence; run_sequence(%r)" % (
        ROOT, str(b))
    subprocess.run([sys.executable, "-c", code], env=env, check=True)
    da, db = torch.load(str(a)), torch.load(str(b))
    assert da["debug"] is False and db["debug"] is True
    assert da["damaged"] == [0] * 5 and db["damaged"] == [0] * 5
    for x, y in zip(da["results"], db["results"]):
        assert torch.equal(x, y)
