"""ctypes binding of include/curvadion.h: the same entry points, argument marshalling only.

Every computation happens inside libcurvadion.so.  Loading fails loudly when the library
has not been built; there is no fallback path.
"""
from __future__ import annotations

import ctypes as C
import os

PKG = os.path.dirname(os.path.abspath(__file__))
# CURVADION_LIB selects another build of the same library (e.g. libcurvadion_debug.so)
LIB_PATH = os.environ.get("CURVADION_LIB") or os.path.join(PKG, "libcurvadion.so")

DION_OK = 0
DION_ERR_INVALID_ARG = 1
DION_ERR_UNSUPPORTED = 2
DION_ERR_ALIGNMENT = 3
DION_ERR_CUDA = 4
DION_ERR_BREAKDOWN = 5
DION_ERR_NONFINITE = 6
DION_ERR_TIMEOUT = 7
DION_ERR_CORRUPT = 8

DION_GATE_ALWAYS = 0
DION_GATE_GLOBAL = 1
DION_GATE_PER_LAYER = 2
DION_GATE_SCHEDULED = 3

DION_DTYPE_FP32 = 0
DION_DTYPE_BF16 = 1

DION_PREC_FP32 = 0
DION_PREC_BF16 = 1
DION_PREC_BF16X3 = 2

DION_MAX_RANK = 512

DION_PHASE_NORMS = 1
DION_PHASE_POWER = 2
DION_PHASE_ORTHO = 3
DION_PHASE_UPDATE = 4

# Every function declared in include/curvadion.h.
EXPORTED = ("dion_plan_create", "dion_step", "dion_get_device_status", "dion_plan_refresh", "dion_step_launch_count",
            "dion_timing_enable", "dion_timing_read", "dion_buffer_norms_noalloc", "dion_plan_destroy",
            "dion_status_string", "dion_abi_version", "dion_plan_enable_host_gradients", "dion_step_host",
            "dion_lr_schedule", "dion_rank_for", "dion_plan_set_wait_limit", "dion_step_phase", "dion_plan_exchange",
            "dion_plan_check_guards", "dion_debug_checks")

DION_ABI_VERSION = 3
DION_NOALLOC_MAX_LAYERS = 256
DION_NOALLOC_MAX_TILES = 65536


class dion_layer(C.Structure):
    _fields_ = [
        ("m", C.c_int64), ("n", C.c_int64), ("r", C.c_int64),
        ("X", C.c_void_p), ("ldx", C.c_int64),
        ("M", C.c_void_p), ("ldm", C.c_int64),
        ("Q", C.c_void_p), ("ldq", C.c_int64),
        ("G", C.c_void_p), ("ldg", C.c_int64),
        ("g_dtype", C.c_int32),
        ("tau", C.c_float),
    ]


class dion_hparams(C.Structure):
    _fields_ = [
        ("mu", C.c_float), ("eta", C.c_float), ("eta_local", C.c_float),
        ("eps_rmmc", C.c_float), ("eps_col", C.c_float), ("tau_global", C.c_float),
        ("gate_mode", C.c_int32), ("period", C.c_int32), ("step", C.c_int64),
        ("weight_decay", C.c_float),
    ]


class DionError(RuntimeError):
    def __init__(self, code: int, what: str = ""):
        self.code = code
        super().__init__(f"{what}: {dion_status_string(code)} ({code})")


_lib = None


def load(path: str = LIB_PATH) -> C.CDLL:
    """Loads libcurvadion.so (built by paper_2512_13728_gb300.build) and declares its signatures."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: build it with `python -m paper_2512_13728_gb300.build`")
    lib = C.CDLL(path)
    P = C.c_void_p
    lib.dion_plan_create.argtypes = [C.POINTER(dion_layer), C.c_int32, C.c_int32, C.POINTER(P)]
    lib.dion_plan_create.restype = C.c_int
    lib.dion_step.argtypes = [P, C.POINTER(dion_hparams), P, P, P, P, P, P]
    lib.dion_step.restype = C.c_int
    lib.dion_plan_enable_host_gradients.argtypes = [P]
    lib.dion_plan_enable_host_gradients.restype = C.c_int
    lib.dion_step_host.argtypes = [P, C.POINTER(dion_hparams), C.POINTER(P), C.POINTER(C.c_int64), P, P, P, P, P, P]
    lib.dion_step_host.restype = C.c_int
    lib.dion_lr_schedule.argtypes = [C.c_int64, C.c_int64, C.c_float, C.c_float, C.c_float]
    lib.dion_lr_schedule.restype = C.c_float
    lib.dion_rank_for.argtypes = [C.c_int64, C.c_int64, C.c_double]
    lib.dion_rank_for.restype = C.c_int64
    lib.dion_get_device_status.argtypes = [P, C.c_int32, C.POINTER(C.c_int32)]
    lib.dion_get_device_status.restype = C.c_int
    lib.dion_plan_refresh.argtypes = [P, P]
    lib.dion_plan_refresh.restype = C.c_int
    lib.dion_step_launch_count.argtypes = [P]
    lib.dion_step_launch_count.restype = C.c_int32
    lib.dion_timing_enable.argtypes = [P, C.c_int32]
    lib.dion_timing_enable.restype = C.c_int
    lib.dion_timing_read.argtypes = [P, C.c_int32, C.POINTER(C.c_float), C.POINTER(C.c_char_p),
                                     C.POINTER(C.c_int32), C.POINTER(C.c_int32)]
    lib.dion_timing_read.restype = C.c_int
    lib.dion_buffer_norms_noalloc.argtypes = [C.POINTER(dion_layer), C.c_int32, P, P, P]
    lib.dion_buffer_norms_noalloc.restype = C.c_int
    lib.dion_step_phase.argtypes = [P, C.c_int32, C.POINTER(dion_hparams), P, P, P, P, P, P]
    lib.dion_step_phase.restype = C.c_int
    lib.dion_plan_exchange.argtypes = [P, C.c_int32, C.POINTER(P), C.POINTER(C.c_int64)]
    lib.dion_plan_exchange.restype = C.c_int
    lib.dion_plan_check_guards.argtypes = [P, C.POINTER(C.c_int32)]
    lib.dion_plan_check_guards.restype = C.c_int
    lib.dion_debug_checks.argtypes = []
    lib.dion_debug_checks.restype = C.c_int32
    lib.dion_plan_set_wait_limit.argtypes = [P, C.c_int64]
    lib.dion_plan_set_wait_limit.restype = C.c_int
    lib.dion_plan_destroy.argtypes = [P]
    lib.dion_plan_destroy.restype = None
    lib.dion_status_string.argtypes = [C.c_int]
    lib.dion_status_string.restype = C.c_char_p
    lib.dion_abi_version.argtypes = []
    lib.dion_abi_version.restype = C.c_int32
    if lib.dion_abi_version() != DION_ABI_VERSION:  # the structs above follow this version's header
        raise ImportError(f"{path} has ABI version {lib.dion_abi_version()}, this binding expects {DION_ABI_VERSION}: "
                          "rebuild it with `python -m paper_2512_13728_gb300.build --force`")
    _lib = lib
    return lib


def dion_status_string(code: int) -> str:
    return load().dion_status_string(int(code)).decode()


def dion_abi_version() -> int:
    return int(load().dion_abi_version())


def dion_plan_create(layers, precision: int) -> int:
    """layers: sequence of dion_layer; returns the opaque plan handle (an int)."""
    arr = (dion_layer * max(len(layers), 1))(*layers)
    out = C.c_void_p()
    st = load().dion_plan_create(arr, len(layers), int(precision), C.byref(out))
    if st != DION_OK:
        raise DionError(st, "dion_plan_create")
    return out.value


def dion_step(plan: int, hp: dion_hparams, prev_norm: int, rmmc_out: int, rmmc_eq1_out, sync_flags_out: int,
              global_flag_out: int, stream: int) -> None:
    """All pointers are device addresses (ints); rmmc_eq1_out may be None."""
    st = load().dion_step(C.c_void_p(plan), C.byref(hp), C.c_void_p(prev_norm), C.c_void_p(rmmc_out),
                          C.c_void_p(rmmc_eq1_out) if rmmc_eq1_out else None, C.c_void_p(sync_flags_out),
                          C.c_void_p(global_flag_out), C.c_void_p(stream) if stream else None)
    if st != DION_OK:
        raise DionError(st, "dion_step")


def dion_step_phase(plan: int, phase: int, hp: dion_hparams, prev_norm: int, rmmc_out: int, rmmc_eq1_out,
                    sync_flags_out: int, global_flag_out: int, stream: int) -> None:
    """One phase (DION_PHASE_*) of a data-parallel step; pointers as in dion_step."""
    st = load().dion_step_phase(C.c_void_p(plan), int(phase), C.byref(hp), C.c_void_p(prev_norm), C.c_void_p(rmmc_out),
                                C.c_void_p(rmmc_eq1_out) if rmmc_eq1_out else None, C.c_void_p(sync_flags_out),
                                C.c_void_p(global_flag_out), C.c_void_p(stream) if stream else None)
    if st != DION_OK:
        raise DionError(st, "dion_step_phase")


def dion_plan_exchange(plan: int, phase: int):
    """(device address, fp32 element count) of the range a worker averages after `phase`."""
    buf, cnt = C.c_void_p(), C.c_int64(0)
    st = load().dion_plan_exchange(C.c_void_p(plan), int(phase), C.byref(buf), C.byref(cnt))
    if st != DION_OK:
        raise DionError(st, "dion_plan_exchange")
    return buf.value or 0, int(cnt.value)


def dion_lr_schedule(step: int, total_steps: int, base_lr: float, warmup_frac: float, warmdown_frac: float) -> float:
    return float(load().dion_lr_schedule(int(step), int(total_steps), float(base_lr), float(warmup_frac),
                                         float(warmdown_frac)))


def dion_rank_for(m: int, n: int, fraction: float) -> int:
    return int(load().dion_rank_for(int(m), int(n), float(fraction)))


def dion_plan_enable_host_gradients(plan: int) -> None:
    st = load().dion_plan_enable_host_gradients(C.c_void_p(plan))
    if st != DION_OK:
        raise DionError(st, "dion_plan_enable_host_gradients")


def dion_step_host(plan: int, hp: dion_hparams, host_G, host_ldg, prev_norm: int, rmmc_out: int, rmmc_eq1_out,
                   sync_flags_out: int, global_flag_out: int, stream: int) -> None:
    """host_G: host addresses (ints) of the layers' gradients, host_ldg: their leading dimensions
    (elements); the other pointers are device addresses as in dion_step."""
    n = max(len(host_G), 1)
    gp = (C.c_void_p * n)(*[C.c_void_p(int(a)) for a in host_G])
    ld = (C.c_int64 * n)(*[int(v) for v in host_ldg])
    st = load().dion_step_host(C.c_void_p(plan), C.byref(hp), gp, ld, C.c_void_p(prev_norm), C.c_void_p(rmmc_out),
                               C.c_void_p(rmmc_eq1_out) if rmmc_eq1_out else None, C.c_void_p(sync_flags_out),
                               C.c_void_p(global_flag_out), C.c_void_p(stream) if stream else None)
    if st != DION_OK:
        raise DionError(st, "dion_step_host")


def dion_get_device_status(plan: int, clear: bool = True) -> int:
    code = C.c_int32(0)
    st = load().dion_get_device_status(C.c_void_p(plan), 1 if clear else 0, C.byref(code))
    if st != DION_OK:
        raise DionError(st, "dion_get_device_status")
    return int(code.value)


def dion_plan_refresh(plan: int, stream: int = 0) -> None:
    st = load().dion_plan_refresh(C.c_void_p(plan), C.c_void_p(stream) if stream else None)
    if st != DION_OK:
        raise DionError(st, "dion_plan_refresh")


def dion_step_launch_count(plan: int) -> int:
    return int(load().dion_step_launch_count(C.c_void_p(plan)))


def dion_timing_enable(plan: int, max_steps: int) -> None:
    st = load().dion_timing_enable(C.c_void_p(plan), int(max_steps))
    if st != DION_OK:
        raise DionError(st, "dion_timing_enable")


def dion_timing_read(plan: int):
    """Returns (steps recorded, [(kernel name, average ms per launch), ...]) in launch order."""
    cap = 64
    ms = (C.c_float * cap)()
    names = (C.c_char_p * cap)()
    count, steps = C.c_int32(0), C.c_int32(0)
    st = load().dion_timing_read(C.c_void_p(plan), cap, ms, names, C.byref(count), C.byref(steps))
    if st != DION_OK:
        raise DionError(st, "dion_timing_read")
    n = min(cap, count.value)
    return steps.value, [((names[i] or b"").decode(), float(ms[i])) for i in range(n)]


def dion_buffer_norms_noalloc(layers, norm_b_out: int, norm_m_out: int, stream: int = 0) -> None:
    """B = M + G in place and ||B||, ||M_{t-1}|| per layer, without allocating (see the header)."""
    arr = (dion_layer * max(len(layers), 1))(*layers)
    st = load().dion_buffer_norms_noalloc(arr, len(layers), C.c_void_p(norm_b_out), C.c_void_p(norm_m_out),
                                          C.c_void_p(stream) if stream else None)
    if st != DION_OK:
        raise DionError(st, "dion_buffer_norms_noalloc")


def dion_plan_check_guards(plan: int) -> int:
    """Number of damaged workspace guard words (0 when no kernel wrote past its region)."""
    out = C.c_int32(0)
    st = load().dion_plan_check_guards(C.c_void_p(plan), C.byref(out))
    if st != DION_OK:
        raise DionError(st, "dion_plan_check_guards")
    return int(out.value)


def dion_debug_checks() -> bool:
    return bool(load().dion_debug_checks())


def dion_plan_set_wait_limit(plan: int, limit_ns: int) -> None:
    """Limit of the update kernel's hand-off waits (<= 0: the default of 2 s); a test hook."""
    st = load().dion_plan_set_wait_limit(C.c_void_p(plan), int(limit_ns))
    if st != DION_OK:
        raise DionError(st, "dion_plan_set_wait_limit")


def dion_plan_destroy(plan: int) -> None:
    if plan:
        load().dion_plan_destroy(C.c_void_p(plan))
