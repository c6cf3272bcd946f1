"""The C-ABI library loads, exports every function include/curvadion.h declares, and rejects
bad arguments on the host (CPU only: no kernel is launched; device pointers are fake and
never dereferenced because validation fails first)."""
import ctypes as C
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "curvadion.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2512_13728_gb300 import build, native

    build.build()
    return native.load()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(dion_[a-z_0-9]+)\s*\(", src)))


def test_header_declares_expected_api():
    from paper_2512_13728_gb300 import native

    assert declared_functions() == sorted(native.EXPORTED)


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_exported_symbols_via_nm(lib):
    out = os.popen(f"nm -D --defined-only {lib._name}").read()
    for name in declared_functions():
        assert re.search(rf"\bT {name}$", out, flags=re.M), name


def test_abi_version_and_status_strings(lib):
    from paper_2512_13728_gb300 import native

    assert native.dion_abi_version() == native.DION_ABI_VERSION == 3
    for code in range(9):
        assert native.dion_status_string(code).startswith("DION_")
    assert "unknown" in native.dion_status_string(99)


def fake_layer(**kw):
    from paper_2512_13728_gb300 import native

    base = dict(m=64, n=48, r=8, X=0x10000, ldx=48, M=0x20000, ldm=48, Q=0x30000, ldq=8, G=0x40000, ldg=48,
                g_dtype=native.DION_DTYPE_BF16, tau=0.5)
    base.update(kw)
    return native.dion_layer(**base)


@pytest.mark.parametrize("kw,code", [
    (dict(r=0), 1), (dict(r=49), 1), (dict(m=0), 1), (dict(n=-1), 1),
    (dict(r=513, m=1024, n=1024, ldx=1024, ldm=1024, ldg=1024, ldq=516), 2),
    (dict(X=0), 1), (dict(G=0), 1), (dict(g_dtype=7), 1), (dict(ldx=40), 1), (dict(ldq=4), 1),
    (dict(X=0x10004), 3), (dict(ldm=50), 3), (dict(ldg=52), 3), (dict(ldq=10), 3),
    (dict(tau=float("nan")), 1),
])
def test_plan_create_rejects_bad_layers(lib, kw, code):
    from paper_2512_13728_gb300 import native

    layers = (native.dion_layer * 1)(fake_layer(**kw))
    out = C.c_void_p(123)
    st = lib.dion_plan_create(layers, 1, native.DION_PREC_FP32, C.byref(out))
    assert st == code
    assert out.value is None  # *out cleared on failure


def test_plan_create_rejects_bad_precision_and_counts(lib):
    from paper_2512_13728_gb300 import native

    layers = (native.dion_layer * 1)(fake_layer())
    out = C.c_void_p()
    assert lib.dion_plan_create(layers, 1, 9, C.byref(out)) == 1
    assert lib.dion_plan_create(layers, -1, 0, C.byref(out)) == 1
    assert lib.dion_plan_create(None, 2, 0, C.byref(out)) == 1
    assert lib.dion_plan_create(layers, 1, 0, None) == 1


def test_step_rejects_null_plan(lib):
    from paper_2512_13728_gb300 import hparams

    hp = hparams()
    assert lib.dion_step(None, C.byref(hp), None, None, None, None, None, None) == 1
    code = C.c_int32()
    assert lib.dion_get_device_status(None, 0, C.byref(code)) == 1
    assert lib.dion_step_launch_count(None) == 0
    assert lib.dion_plan_enable_host_gradients(None) == 1
    assert lib.dion_step_host(None, C.byref(hp), None, None, None, None, None, None, None, None) == 1
    lib.dion_plan_destroy(None)  # no-op


def test_hparams_struct_layout():
    from paper_2512_13728_gb300 import native

    assert C.sizeof(native.dion_hparams) == 48
    assert native.dion_hparams.weight_decay.offset == 40


@pytest.mark.parametrize("T,wu,wd", [(3000, 0.01, 0.2), (3000, 0.01, 0.1), (100, 0.0, 0.5), (50, 0.01, 0.0),
                                     (8, 0.5, 0.5), (1, 0.0, 1.0), (50, 0.1, 0.1)])
def test_lr_schedule_matches_oracle(lib, T, wu, wd):
    """The library's host-side schedule (fp32 result) against the oracle's definition."""
    import numpy as np

    import oracle.curvadion as oc
    from paper_2512_13728_gb300 import native

    for t in list(range(-1, min(T, 60) + 2)) + list(range(max(1, T - 60), T + 3)):
        want = np.float32(oc.lr_schedule(t, T, float(np.float32(0.02)), float(np.float32(wu)), float(np.float32(wd))))
        assert native.dion_lr_schedule(t, T, 0.02, wu, wd) == pytest.approx(float(want), rel=2e-7, abs=0.0), t


def test_lr_schedule_rejects_bad_arguments(lib):
    import math

    from paper_2512_13728_gb300 import native

    assert math.isnan(native.dion_lr_schedule(1, 0, 0.02, 0.01, 0.1))
    assert math.isnan(native.dion_lr_schedule(1, 100, 0.02, -0.1, 0.1))
    assert math.isnan(native.dion_lr_schedule(1, 100, 0.02, 0.6, 0.6))
    assert math.isnan(native.dion_lr_schedule(1, 100, 0.02, 0.01, float("nan")))


@pytest.mark.parametrize("m,n,f", [(768, 3072, 0.125), (2048, 8192, 0.125), (100, 100, 0.125), (1, 5, 0.125),
                                   (64, 64, 1.0), (4096, 1024, 1 / 16), (768, 768, 0.25), (3, 1000, 0.3)])
def test_rank_for_matches_oracle(lib, m, n, f):
    import oracle.curvadion as oc
    from paper_2512_13728_gb300 import native

    assert native.dion_rank_for(m, n, f) == oc.rank_for(m, n, f)


def test_rank_for_rejects_bad_arguments(lib):
    from paper_2512_13728_gb300 import native

    assert native.dion_rank_for(0, 5, 0.1) == 0
    assert native.dion_rank_for(5, 5, 0.0) == 0
    assert native.dion_rank_for(5, 5, 1.5) == 0


def test_wait_limit_rejects_null_plan(lib):
    from paper_2512_13728_gb300 import native

    assert lib.dion_plan_set_wait_limit(None, C.c_int64(5)) == native.DION_ERR_INVALID_ARG


def test_phase_entry_points_reject_bad_arguments(lib):
    from paper_2512_13728_gb300 import native

    hp = native.dion_hparams(mu=0.95, eta=0.01, eta_local=0.01, eps_rmmc=1e-8, eps_col=1e-8, tau_global=0.5,
                             gate_mode=0, period=1, step=1)
    assert lib.dion_step_phase(None, native.DION_PHASE_NORMS, C.byref(hp), None, None, None, None, None,
                               None) == native.DION_ERR_INVALID_ARG
    buf, cnt = C.c_void_p(), C.c_int64(0)
    assert lib.dion_plan_exchange(None, native.DION_PHASE_POWER, C.byref(buf), C.byref(cnt)) == \
        native.DION_ERR_INVALID_ARG


def test_guard_entry_points(lib):
    from paper_2512_13728_gb300 import native

    out = C.c_int32(0)
    assert lib.dion_plan_check_guards(None, C.byref(out)) == native.DION_ERR_INVALID_ARG
    assert lib.dion_debug_checks() == 0  # the default build has no debug checks


def test_debug_build_reports_its_checks():
    """The DION_DEBUG_CHECKS variant builds from the same sources and says so (loaded in a child
    process, so this process keeps the default library)."""
    import subprocess
    import sys

    from paper_2512_13728_gb300 import build

    path = build.build(debug=True)
    code = ("import ctypes; l = ctypes.CDLL(%r); l.dion_debug_checks.restype = ctypes.c_int32; "
            "print(l.dion_debug_checks())") % path
    out = subprocess.run([sys.executable, "-c", code], stdout=subprocess.PIPE, text=True, check=True).stdout
    assert out.strip() == "1"
