"""Algorithm 2 with two data-parallel ranks on CPU (gloo, world size 2): each rank holds one
worker's state and gradients and exchanges only what the algorithm exchanges (AllReduce_max of
the per-layer RMMC, AllReduce_DP of P and of R on a sync), with the oracle's per-worker
arithmetic in between; after a run mixing sync and local steps both ranks match the
single-process W-worker emulation ``curvadion_step_dp``."""
import os
import socket
import sys

import numpy as np
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SHAPES = [(24, 16), (16, 40)]
RANKS = [4, 3]
STEPS = 6


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _init(w):
    g = np.random.default_rng(100)  # the same starting point on every worker
    out = []
    for (m, n), r in zip(SHAPES, RANKS):
        q = g.standard_normal((n, r))
        out.append(dict(X=g.standard_normal((m, n)), M=np.zeros((m, n)), Q=q / np.linalg.norm(q, axis=0)))
    return out


def _grad(w, t, l):
    g = np.random.default_rng(1000 * w + 10 * t + l)
    scale = 5.0 if t == 4 and w == 1 else 1.0  # a spike on worker 1 at step 4
    return scale * g.standard_normal(SHAPES[l])


def _hp(oc):
    return oc.HParams(gate_mode=oc.GATE_GLOBAL, tau_global=0.5, weight_decay=0.01)


def _rank_main(rank, world, port, out):
    import torch
    import torch.distributed as dist

    sys.path.insert(0, ROOT)
    import oracle.curvadion as oc

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        hp = _hp(oc)
        st = _init(rank)
        prev = np.zeros(len(SHAPES))
        syncs = []
        for t in range(1, STEPS + 1):
            G = [_grad(rank, t, l) for l in range(len(SHAPES))]
            B = [oc.form_buffer(st[l]["M"], G[l]) for l in range(len(SHAPES))]
            nb = np.array([oc.frobenius_norm(b) for b in B])
            rm = np.array([oc.rmmc_alg2(nb[l], prev[l], hp.eps_rmmc) for l in range(len(SHAPES))])
            prev = nb
            rmax = torch.tensor(rm)
            dist.all_reduce(rmax, op=dist.ReduceOp.MAX)  # AllReduce_max
            _, gflag, active = oc.gate(rmax.numpy(), [0.5] * len(SHAPES), hp.tau_global, hp.gate_mode, t, hp.period)
            syncs.append(bool(gflag))
            for l, (m, n) in enumerate(SHAPES):
                if active[l]:
                    P = torch.tensor(oc.power_iter(B[l], st[l]["Q"]))
                    dist.all_reduce(P)  # AllReduce_DP (mean)
                    P = oc.orthogonalize(P.numpy() / world)
                    R = torch.tensor(B[l].T @ P)
                    dist.all_reduce(R)
                    R = R.numpy() / world
                    st[l]["M"] = B[l] - (1.0 - hp.mu) * (P @ R.T)
                    st[l]["Q"] = oc.column_normalize(R, hp.eps_col)
                    st[l]["X"] = (oc.decay_parameters(st[l]["X"], hp.eta, hp.weight_decay)
                                  - hp.eta * np.sqrt(m / n) * (P @ st[l]["Q"].T))
                else:
                    st[l]["M"], st[l]["X"] = oc.local_update(B[l], G[l], st[l]["X"], hp.eta_local, hp.weight_decay)
        out[rank] = ([{k: v.copy() for k, v in d.items()} for d in st], syncs)
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_ranks_match_the_w_worker_emulation():
    sys.path.insert(0, ROOT)
    import oracle.curvadion as oc

    world, port = 2, _free_port()
    with mp.get_context("spawn").Manager() as mgr:  # no fork of a threaded process
        out = mgr.dict()
        mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
        got = dict(out)
    hp = _hp(oc)
    workers = [[oc.LayerState(X=d["X"], M=d["M"], Q=d["Q"], tau=0.5) for d in _init(w)] for w in range(world)]
    prev = [np.zeros(len(SHAPES)) for _ in range(world)]
    syncs = []
    for t in range(1, STEPS + 1):
        o = oc.curvadion_step_dp(workers, [[_grad(w, t, l) for l in range(len(SHAPES))] for w in range(world)],
                                 prev, hp, t)
        workers, prev = o.workers, o.prev_norm
        syncs.append(o.global_flag)
    assert any(syncs) and not all(syncs)  # the run mixes sync and local steps
    for w in range(world):
        st, rank_syncs = got[w]
        assert rank_syncs == syncs
        for l in range(len(SHAPES)):
            for f in ("X", "M", "Q"):
                assert np.allclose(st[l][f], getattr(workers[w][l], f), rtol=0, atol=1e-12), (w, l, f)
    assert not np.allclose(got[0][0][0]["X"], got[1][0][0]["X"])  # local steps let the workers drift
