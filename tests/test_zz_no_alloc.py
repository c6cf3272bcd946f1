"""dion_buffer_norms_noalloc against the existing entry point (dion_step), on the GPU.

The allocation-free entry point exists for callers that cannot call cudaMalloc (a framework
whose allocator has reserved all device memory up front, or a latency-critical loop where an
allocation would synchronize the device).  It performs the buffer step B = M + G in place and
returns ||B|| and ||M_{t-1}|| per layer.  A dion_step whose layers all take the local branch
(per-layer gate, tau = inf) performs the same buffer step and records ||B|| in prev_norm, so
two calls in a row of each must agree: M bit for bit, the norms to the RMMC tolerance.
This file is collected last on purpose and needs nothing from the other test files.
"""
import ctypes as C
import math

import pytest
import torch

pytestmark = pytest.mark.gpu

RTOL = 1e-5  # the RMMC tolerance of the parity tests (fp32 partial sums folded into fp64)
# (2048, 4096) is 128 tiles of 16 rows, so the reduction's lanes take several tiles each
SHAPES = [(200, 136, "bf16"), (136, 200, "fp32"), (67, 33, "bf16"), (1, 5, "bf16"), (300, 1024, "bf16"),
          (2048, 4096, "bf16")]


@pytest.fixture(scope="module")
def cd():
    from paper_2512_13728_gb300 import build

    build.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    import paper_2512_13728_gb300 as pkg

    return pkg


def make(shapes, seed=3):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    X, M, Q, G = [], [], [], []
    for m, n, dt in shapes:
        ld = (n + 7) // 8 * 8  # 16-byte rows for fp32 and bf16
        X.append(torch.randn(m, ld, device="cuda", generator=g)[:, :n])
        M.append(torch.randn(m, ld, device="cuda", generator=g)[:, :n])
        Q.append(torch.randn(n, 8, device="cuda", generator=g)[:, :1])  # r = 1, 16-byte rows
        gg = torch.randn(m, ld, device="cuda", generator=g) * 0.1
        G.append((gg.to(torch.bfloat16) if dt == "bf16" else gg)[:, :n])
    return X, M, Q, G


def test_noalloc_matches_dion_step_two_calls(cd):
    X, M, Q, G = make(SHAPES)
    M_b = []  # the no-alloc path works on its own copy of M, with the same 16-byte row padding
    for m in M:
        buf = torch.empty(m.shape[0], m.stride(0), device="cuda")[:, : m.shape[1]]
        buf.copy_(m)
        M_b.append(buf)
    plan = cd.Plan(X, M, Q, G, [math.inf] * len(SHAPES), cd.DION_PREC_FP32)
    layers_b = [cd.native.dion_layer(m=x.shape[0], n=x.shape[1], r=1, X=0, ldx=0, M=mb.data_ptr(), ldm=mb.stride(0),
                                     Q=0, ldq=0, G=g.data_ptr(), ldg=g.stride(0),
                                     g_dtype=cd.DION_DTYPE_BF16 if g.dtype == torch.bfloat16 else cd.DION_DTYPE_FP32,
                                     tau=0.0)
                for x, mb, g in zip(X, M_b, G)]
    L = len(SHAPES)
    nb = torch.zeros(L, dtype=torch.float64, device="cuda")
    nm = torch.zeros(L, dtype=torch.float64, device="cuda")
    prev = []
    try:
        for t in (1, 2):
            plan.step(cd.hparams(step=t, gate_mode=cd.DION_GATE_PER_LAYER, tau_global=math.inf))
            cd.native.dion_buffer_norms_noalloc(layers_b, nb.data_ptr(), nm.data_ptr(),
                                                torch.cuda.current_stream().cuda_stream)
            torch.cuda.synchronize()
            assert plan.device_status() == 0
            assert not plan.flags[:L].any()  # every layer took the local branch: M = B
            for ma, mb in zip(M, M_b):
                assert torch.equal(ma, mb)
            want_b = plan.prev_norm[:L]
            assert torch.allclose(nb, want_b, rtol=RTOL, atol=0.0), (t, nb, want_b)
            if prev:  # ||M_{t-1}|| is the previous call's ||B||
                assert torch.allclose(nm, prev[-1], rtol=RTOL, atol=0.0)
            prev.append(want_b.clone())
    finally:
        plan.close()


def test_noalloc_rejects_sizes_beyond_its_scratch(cd):
    X, M, Q, G = make(SHAPES[:1])
    lay = cd.native.dion_layer(m=M[0].shape[0], n=M[0].shape[1], r=1, X=0, ldx=0, M=M[0].data_ptr(),
                               ldm=M[0].stride(0), Q=0, ldq=0, G=G[0].data_ptr(), ldg=G[0].stride(0),
                               g_dtype=cd.DION_DTYPE_BF16, tau=0.0)
    lib = cd.native.load()
    nb = torch.zeros(cd.native.DION_NOALLOC_MAX_LAYERS + 1, dtype=torch.float64, device="cuda")
    too_many = (cd.native.dion_layer * (cd.native.DION_NOALLOC_MAX_LAYERS + 1))(
        *([lay] * (cd.native.DION_NOALLOC_MAX_LAYERS + 1)))
    st = lib.dion_buffer_norms_noalloc(too_many, cd.native.DION_NOALLOC_MAX_LAYERS + 1, C.c_void_p(nb.data_ptr()),
                                       C.c_void_p(nb.data_ptr()), None)
    assert st == cd.native.DION_ERR_UNSUPPORTED
    # more tiles than the scratch holds: a 70000 x 65536 layer is 70000 one-row tiles.  The sizes
    # are checked before any device work, so the small buffer behind the pointers is never read.
    big = cd.native.dion_layer(m=70000, n=65536, r=1, X=0, ldx=0, M=M[0].data_ptr(), ldm=65536, Q=0, ldq=0,
                               G=G[0].data_ptr(), ldg=65536, g_dtype=cd.DION_DTYPE_BF16, tau=0.0)
    before = M[0].clone()
    st = lib.dion_buffer_norms_noalloc((cd.native.dion_layer * 1)(big), 1, C.c_void_p(nb.data_ptr()),
                                       C.c_void_p(nb.data_ptr()), None)
    assert st == cd.native.DION_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert torch.equal(M[0], before)
