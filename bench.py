"""Benchmark of one full-model CurvaDion optimizer step on synthetic GPT-shaped layer stacks.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--workload NAME] [--precision bf16|bf16x3|fp32] [--no-cpu-baseline]

Prints ONE JSON line (rank 0).  A step is dion_step over every layer of the workload (all
hot-path kernels), with inputs resident in HBM; each step moves far more than the 129 MB
L2 (36 GB for the 1.3B-shaped stack), so no explicit L2 flush is needed between steps.
`--impl reference` times the fp64 CPU oracle on the host cores instead (bounded sample).
Under torchrun (N > 1) every rank runs an independent replica of the full step (the path
has no data-path exchange on one GPU per replica) and rank 0 reports the max over ranks.
"""
from __future__ import annotations

import argparse
import csv
import hashlib
import io
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "ms per full-model Dion+RMMC step (160M/1.3B shapes); % of HBM roofline"
UNIT = "ms/step"
DEFAULT_WORKLOAD = "gpt1p3b_stack_r512"
PREC = {"fp32": 0, "bf16": 1, "bf16x3": 2}
DTYPE_NAME = {"fp32": "f32", "bf16": "bf16", "bf16x3": "bf16x3"}


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return dict(hbm=p["hbm_gbs"], bf16=p["bf16_tflops"], bf16_sust=p["bf16_tflops_sustained"],
                    sm_mhz=p.get("sm_max_mhz", 2070.0), source="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sust=1700.0, sm_mhz=2070.0, source="fallback")


def load_tf32_peak():
    """cuBLAS tf32 throughput measured on this machine's GB300 (`bench.py --tf32-peak`), else half of
    the bf16 peak (the nominal ratio)."""
    path = os.path.join(ROOT, "profiles", "tf32_peak.json")
    if os.path.exists(path):
        with open(path) as f:
            return float(json.load(f)["tf32_tflops"]), "measured"
    return load_peaks()["bf16"] / 2, "half of bf16"


def sources_hash(names) -> str:
    """Hash of the listed files under the package's csrc/ (the translation unit of one kernel and
    its host-side schedule), so a stored ncu counter stays valid until that code changes."""
    h = hashlib.sha1()
    d = os.path.join(ROOT, "paper_2512_13728_gb300", "csrc")
    for name in sorted(names):
        with open(os.path.join(d, name), "rb") as f:
            h.update(name.encode() + f.read())
    with open(os.path.join(ROOT, "include", "curvadion.h"), "rb") as f:
        h.update(f.read())
    return h.hexdigest()[:12]


# ------------------------------------------------------------------ algorithmic work ---

def kernel_work(name: str, w, prec: str, gate: str = "always", wt=None, peaks=None):
    """(bound, algorithmic units per launch, unit) for one kernel of the step.  wt[l] is the
    fraction of the timed steps in which layer l took the Dion branch (all 1 with --gate always);
    kernels that run only on syncing layers count those layers' work by it.  Bytes count each
    compulsory read and write once; flops count 2 per multiply-add.  With `peaks`, a bf16
    contraction (B Q, B^T P, the update) is held to whichever of its two rooflines takes longer:
    its bytes at the HBM copy rate or its tensor flops at the sustained bf16 rate (BF16X3 issues
    three products per multiply-add)."""
    base_work = _kernel_work(name, w, prec, gate, wt)
    if peaks is None or base_work[0] != "hbm":
        return base_work
    base = name.rstrip("0123456789")
    ranks = w.ranks()
    wts = [1.0] * len(w.shapes) if wt is None else list(wt)
    mnr = sum(m * n * r * wts[l] for l, ((m, n), r) in enumerate(zip(w.shapes, ranks)))
    prods = 3 if prec == "bf16x3" else 1
    flops = {"tc_bq": 2 * mnr, "tc_form_bq": 2 * mnr, "tc_btp": 2 * mnr, "tc_update": 4 * mnr}.get(base)
    if flops is None:
        return base_work
    t_hbm = base_work[1] / (peaks["hbm"] * 1e9)
    t_tensor = prods * flops / (peaks["bf16_sust"] * 1e12)
    return ("tensor", prods * flops, "flop") if t_tensor > t_hbm else base_work


def _kernel_work(name: str, w, prec: str, gate: str = "always", wt=None):
    gsz = 2 if w.g_dtype == "bf16" else 4
    ranks = w.ranks()
    L = len(w.shapes)
    wt = [1.0] * L if wt is None else list(wt)

    def tot(f, act=True):  # sum over layers of f(m, n, r), weighted by activity
        return sum(f(m, n, r) * (wt[l] if act else 1.0) for l, ((m, n), r) in enumerate(zip(w.shapes, ranks)))

    mn_all = tot(lambda m, n, r: m * n, act=False)
    mn = tot(lambda m, n, r: m * n)
    mn_loc = mn_all - mn
    mnr = tot(lambda m, n, r: m * n * r)
    mr2 = tot(lambda m, n, r: m * r * r)
    mrr1 = tot(lambda m, n, r: m * r * (r + 1))  # a symmetric Gram or a triangular solve: 2 m r (r + 1) / 2
    r3 = tot(lambda m, n, r: r ** 3)
    nr = tot(lambda m, n, r: n * r)
    mr = tot(lambda m, n, r: m * r)
    # the bf16 copy of B the tensor-core contractions read (its two halves with split operands)
    bh = {"bf16": 2, "bf16x3": 4}.get(prec, 0)
    hl = 2 if prec == "bf16x3" else 1  # bf16 copies of P, R, Q: one, or a high and a low half
    # tensor-core mode with bf16 G: in DION_GATE_ALWAYS the buffer pass leaves M_{t-1} in place
    # and the update forms B = M + G itself (it reads G); in the gated modes the norms pass
    # writes B into M first, and neither the fused B Q kernel nor the update reads G
    fused = prec == "bf16" and w.g_dtype == "bf16"
    b_in_m = fused and gate != "always"
    deferred = fused and not b_in_m
    # BF16X3 in a gated mode: the buffer pass writes B alone; split_b writes the halves of the
    # syncing layers' B after the gate
    x3_split = prec == "bf16x3" and gate != "always"
    table = {
        # CUDA-core path (form_b runs on every layer before the gate)
        "form_b": ("hbm", mn_all * (4 + gsz + (0 if fused else 4) + (0 if x3_split else bh)), "B"),
        "split_b": ("hbm", mn * 8, "B") if x3_split else ("latency", 0, ""),  # read B; write hi, lo
        "gemm_bq": ("alu", 2 * mnr, "flop"),
        "gemm_gram": ("alu", 2 * mr2, "flop"),
        "chol_inv": ("alu", 2 * r3 / 3, "flop"),
        "gemm_trsm": ("alu", 2 * mr2, "flop"),
        "gemm_btp": ("alu", 2 * mnr, "flop"),
        "colnorm": ("hbm", nr * 8, "B"),
        "update": ("alu", 4 * mnr, "flop") if prec == "fp32" else ("hbm", mn * 16, "B"),
        # local layers: read X, G; write X (M already holds B)
        "local": ("hbm", mn_loc * (8 + gsz), "B"),
        # tensor-core path
        "tc_bq": ("hbm", mn * bh + nr * 2 * hl + mr * 8, "B"),  # Bh (and Bl), bf16 Q; P and P^T fp32
        # buffer pass fused into B Q (bf16 G): read M (and G unless B is already in M); write Bh,
        # P and P^T fp32
        "tc_form_bq": ("hbm", mn * (4 + (0 if b_in_m else gsz) + 2) + mr * 8, "B"),
        # gated modes: the norms pass reads M, G and writes B into M on every layer (and runs
        # the gate in its last block)
        "norms_gate": ("hbm", mn_all * (4 + gsz + 4), "B"),
        "tc_btp": ("hbm", mn * bh + mr * 2 * hl + nr * (4 + 2 * hl), "B"),  # Bh (Bl), bf16 P; R fp32, bf16
        "tc_update": ("hbm", mn * (16 + (gsz if deferred else 0)), "B"),
        # tf32 tensor work: BF16X3 issues three products (hi.hi + hi.lo + lo.hi) per multiply-add
        "tc_gram": ("tf32", mrr1 * (3 if prec == "bf16x3" else 1), "flop"),
        "tc_trsm": ("tf32", mrr1 * (3 if prec == "bf16x3" else 1), "flop"),
    }
    # Orthogonalize's launches carry their pass: passes 0 and 1 run the Gram and the solve on
    # every synchronizing layer; pass 1's factor is usually the first-order one and pass 2 runs
    # only after a shifted retry, so those count as latency
    base = name.rstrip("0123456789")
    npass = int(name[len(base):]) if len(base) < len(name) else 0
    if npass == 2 or (base == "chol_inv" and npass == 1):
        return ("latency", 0, "")
    return table.get(base, ("latency", 0, ""))


def step_bytes(w, prec, gate: str = "always", wt=None):
    """Bytes one step moves by design (the planned passes) and the compulsory floor (read M, G,
    X; write M, X: 18 B/element with bf16 G, on either branch), with layer l syncing in a
    fraction wt[l] of the steps."""
    gsz = 2 if w.g_dtype == "bf16" else 4
    L = len(w.shapes)
    wt = [1.0] * L if wt is None else list(wt)
    mn_all = sum(m * n for m, n in w.shapes)
    mn = sum(m * n * wt[l] for l, (m, n) in enumerate(w.shapes))
    mn_loc = mn_all - mn
    fused = prec == "bf16" and w.g_dtype == "bf16"
    if prec == "fp32":  # form_b 12 (+4 with fp32 G), B Q and B^T P read B 4 + 4, update 16
        planned = mn_all * (4 + gsz + 4) + mn * (4 + 4 + 16)
    elif prec == "bf16x3" and gate == "always":  # form_b writes M, Bh, Bl; B Q, B^T P read both halves, update 16
        planned = mn_all * (4 + gsz + 4 + 4) + mn * (4 + 4 + 16)
    elif prec == "bf16x3":  # form_b writes M; synced: split_b 8, B Q and B^T P 4 + 4, update 16
        planned = mn_all * (4 + gsz + 4) + mn * (8 + 4 + 4 + 16)
    elif fused and gate == "always":  # buffer pass fused with B Q 8, the Bh read of B^T P 2, update 18
        planned = mn_all * ((4 + gsz + 2) + 2 + (16 + gsz))
    elif fused:  # norms pass 10 on every layer; synced: fused B Q 6, Bh read 2, update 16
        planned = mn_all * (4 + gsz + 4) + mn * (6 + 2 + 16)
    else:  # form_b 14 with fp32 G, Bh read of B Q and B^T P 2 + 2, update 16
        planned = mn_all * (4 + gsz + 4 + 2) + mn * (2 + 2 + 16)
    planned += mn_loc * (8 + gsz)  # local branch: read X, G; write X
    compulsory = mn_all * (4 + gsz + 4 + 4 + 4)  # read M, G, X; write M, X
    return planned, compulsory


def make_gradient_sequence(wl, w, dtype, dev, steps):
    """One flat device tensor per step t in `steps` holding every layer's G_t (row-major, layer
    after layer)."""
    import torch

    out = []
    for t in steps:
        out.append(torch.cat([wl.gradient(w, l, t, dev).to(dtype).reshape(-1) for l in range(w.num_layers)]))
    return out


def layer_views(flat, w):
    """Each layer's m x n gradient as a view of the flat buffer."""
    views, off = [], 0
    for m, n in w.shapes:
        views.append(flat[off: off + m * n].view(m, n))
        off += m * n
    return views


def replay_sync_pattern(cd, wl, w, prec_code, gate_code, tau, t0, warmup, steps, seq, dev):
    """Which layers took the Dion branch in each timed step, from an untimed replay of the same
    run (same seeded initial state, gradient sequence and hyper-parameters; a plan's steps are
    deterministic, so it reaches the same decisions).  Returns per-layer fractions of the timed
    steps and the number of syncing layers in each."""
    X, M, Q = [], [], []
    for l in range(w.num_layers):
        x0, m0, q0 = wl.init_layer(w, l, dev)
        X.append(x0); M.append(m0); Q.append(q0)
    gflat = seq[0].clone()
    L = w.num_layers
    plan = cd.Plan(X, M, Q, layer_views(gflat, w), [tau] * L, prec_code)
    counts, per_step = [0] * L, []
    try:
        for i in range(warmup + steps):
            gflat.copy_(seq[i])
            plan.step(cd.hparams(step=t0 + i, gate_mode=gate_code, tau_global=tau))
            if i < warmup:
                continue
            if gate_code == cd.DION_GATE_GLOBAL:
                act = [bool(plan.global_flag[0].item())] * L
            else:
                act = plan.flags[:L].cpu().numpy().astype(bool).tolist()
            per_step.append(int(sum(act)))
            for l in range(L):
                counts[l] += int(act[l])
    finally:
        plan.close()
    return [c / steps for c in counts], per_step


# ---------------------------------------------------------------------------- clocks ---

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.proc = None
        self.gpu_id = gpu_id

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", self.gpu_id, f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (FileNotFoundError, OSError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=10)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = [r for r in csv.reader(io.StringIO(out)) if len(r) >= 7]
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            try:
                sm.append(float(r[0]))
                mx.append(float(r[1]))
            except ValueError:
                continue
            for k, v in zip(names, r[3:7]):
                if v.strip().lower() == "active":
                    reasons.add(k)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# --------------------------------------------------------------------- our GPU arm ---

def max_over_ranks(value: float, world: int, device) -> float:
    """The slowest replica's time: every rank contributes its own, every rank gets the max
    (NCCL on the GPU in the bench; any backend whose tensors live on `device`)."""
    if world <= 1:
        return float(value)
    import torch
    import torch.distributed as dist

    t = torch.tensor([float(value)], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def kernel_frac(k, peaks):
    """{"bound", "frac"} of one kernel's measured time against its roofline (HBM copy, bf16 or
    tf32 tensor throughput), or {} for latency-bound kernels."""
    if k["ms"] <= 0 or not k["units"]:
        return {}
    rate = k["units"] / (k["ms"] * 1e-3)
    if k["bound"] == "hbm":
        return {"bound": "hbm", "frac": round(rate / 1e9 / peaks["hbm"], 4)}
    if k["bound"] == "tensor":
        return {"bound": "bf16", "frac": round(rate / 1e12 / peaks["bf16_sust"], 4)}
    if k["bound"] == "tf32":
        return {"bound": "tf32", "frac": round(rate / 1e12 / load_tf32_peak()[0], 4)}
    if k["bound"] == "alu":
        return {"bound": "fp32 FFMA", "frac": round(rate / 1e12 / (152 * 128 * 2 * peaks["sm_mhz"] * 1e6 / 1e12), 4)}
    return {}


def run_ours(args, rank, world, local_rank):
    import torch

    import paper_2512_13728_gb300 as cd
    import workloads as wl
    from paper_2512_13728_gb300 import build as cdbuild

    if rank == 0 or world == 1:
        cdbuild.build()
    if world > 1:
        import torch.distributed as dist

        dist.barrier()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    w = wl.WORKLOADS[args.workload]
    prec = args.precision
    gdt = torch.bfloat16 if w.g_dtype == "bf16" else torch.float32

    # Gated runs follow the workload's gradient sequence G_t (the branch each layer takes depends
    # on it); every layer's G is a view of one flat buffer, and step t's gradients are copied into
    # it before the step, outside the step's timed interval.  With DION_GATE_ALWAYS every layer
    # does the same work whatever G holds, so G_1 stays in place and the steps run back to back.
    grad_seq = args.gate != "always"
    X, M, Q = [], [], []
    for l in range(w.num_layers):
        x0, m0, q0 = wl.init_layer(w, l, dev)
        X.append(x0); M.append(m0); Q.append(q0)
    seq = make_gradient_sequence(wl, w, gdt, dev, range(args.t0, args.t0 + (args.warmup + args.steps if grad_seq
                                                                              else 1)))
    gflat = seq[0].clone() if grad_seq else seq.pop()
    G = layer_views(gflat, w)
    torch.cuda.synchronize()
    plan = cd.Plan(X, M, Q, G, [args.tau] * w.num_layers, PREC[prec])
    gate = {"always": cd.DION_GATE_ALWAYS, "global": cd.DION_GATE_GLOBAL, "per_layer": cd.DION_GATE_PER_LAYER}[args.gate]
    stream = torch.cuda.current_stream(dev)
    t = args.t0 - 1

    def one_step():
        nonlocal t
        t += 1
        plan.step(cd.hparams(step=t, gate_mode=gate, tau_global=args.tau), stream=stream.cuda_stream)

    def load_gradients(i):
        if grad_seq:
            gflat.copy_(seq[i], non_blocking=True)

    for i in range(args.warmup):
        load_gradients(i)
        one_step()
    torch.cuda.synchronize()
    if plan.device_status() != 0:
        raise RuntimeError("device status after warm-up: " + cd.native.dion_status_string(plan.device_status()))

    # --graph: one step captured into a CUDA graph (every kernel of dion_step is enqueued without
    # a host sync or an allocation, so the call can be captured) and replayed in the timed region;
    # the per-kernel breakdown then comes from eager steps timed after it
    graph = None
    if args.graph:
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            plan.step(cd.hparams(step=t + 1, gate_mode=gate, tau_global=args.tau))
        torch.cuda.synchronize()
    # ---- timed region (device-resident inputs) ----
    if graph is None:
        cd.native.dion_timing_enable(plan.handle, args.steps)
    sampler = None
    if rank == 0:
        props = torch.cuda.get_device_properties(dev)
        uuid = getattr(props, "uuid", None)
        gid = f"GPU-{uuid}" if uuid is not None and not str(uuid).startswith("GPU-") else (str(uuid) if uuid else
                                                                                           str(local_rank))
        sampler = ClockSampler(gid)
        sampler.start()
        time.sleep(0.3)
    if world > 1:
        import torch.distributed as dist

        dist.barrier()
    torch.cuda.synchronize()
    if grad_seq:  # one event pair per step; the gradient copies fall between them
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
        for i in range(args.steps):
            load_gradients(args.warmup + i)
            evs[i][0].record(stream)
            one_step()
            evs[i][1].record(stream)
    elif graph is not None:  # the same step replayed from a CUDA graph (launch overhead removed)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            graph.replay()
        e1.record(stream)
    else:
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            one_step()
        e1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clocks = sampler.stop() if sampler else None
    ms_total = sum(a.elapsed_time(b) for a, b in evs) if grad_seq else e0.elapsed_time(e1)
    if graph is not None:  # per-kernel times from eager steps
        cd.native.dion_timing_enable(plan.handle, args.steps)
        for _ in range(args.steps):
            one_step()
        torch.cuda.synchronize()
    nsteps_timed, ktimes = cd.native.dion_timing_read(plan.handle)
    cd.native.dion_timing_enable(plan.handle, 0)
    ms_total = max_over_ranks(ms_total, world, dev)
    if plan.device_status() != 0:
        raise RuntimeError("device status after timed steps is not OK")
    ms_step = ms_total / args.steps

    # ---- end to end: H2D of the step's gradient from pinned host memory + step + D2H of results ----
    # Through the C ABI's host-gradient entry point: each step copies every layer's G_t from
    # pinned host memory into one of the plan's two device buffers (on the plan's copy stream,
    # overlapping the previous step's kernels), runs the step behind the copies, and reads the
    # step's RMMC values and flags back into pinned host memory.
    host_G = [g.cpu().pin_memory() for g in G]
    host_out = torch.empty(w.num_layers * 9 + 1, dtype=torch.uint8).pin_memory()
    h2d = sum(g.numel() * g.element_size() for g in host_G)
    d2h = plan.rmmc[: w.num_layers].numel() * 8 + w.num_layers + 1
    e_steps = max(1, min(args.steps, 10))
    plan.enable_host_gradients()

    def e2e_step():
        nonlocal t
        t += 1
        plan.step_host(cd.hparams(step=t, gate_mode=gate, tau_global=args.tau), host_G, stream=stream.cuda_stream)
        host_out[: 8 * w.num_layers].copy_(plan.rmmc[: w.num_layers].view(torch.uint8), non_blocking=True)
        host_out[8 * w.num_layers: 9 * w.num_layers].copy_(plan.flags[: w.num_layers], non_blocking=True)
        host_out[9 * w.num_layers:].copy_(plan.global_flag, non_blocking=True)

    for _ in range(max(2, args.warmup)):  # first use of the pinned pages and buffers stays untimed
        e2e_step()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    # three repetitions of e_steps steps, the median reported: the host side of the copies is
    # shared with whatever else the machine runs
    reps = []
    for _ in range(3):
        f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        f0.record(stream)
        for _ in range(e_steps):
            e2e_step()
        f1.record(stream)
        torch.cuda.synchronize()
        reps.append(f0.elapsed_time(f1) / e_steps)
    e2e_ms = sorted(reps)[1]
    e2e_ms = max_over_ranks(e2e_ms, world, dev)
    launches = plan.launches_per_step()
    plan.close()
    if rank != 0:
        return None
    wt, sync_per_step = None, None
    if grad_seq:
        del X, M, Q, G, gflat, host_G
        torch.cuda.empty_cache()
        wt, sync_per_step = replay_sync_pattern(cd, wl, w, PREC[prec], gate, args.tau, args.t0, args.warmup,
                                                args.steps, seq, dev)

    peaks = load_peaks()
    kern = []
    for name, ms in ktimes:
        bound, units, unit = kernel_work(name, w, prec, args.gate, wt, peaks)
        kern.append(dict(name=name, ms=ms, bound=bound, units=units, unit=unit))
    dom = max(kern, key=lambda k: k["ms"]) if kern else None
    roofline = None
    if dom is not None:
        if dom["bound"] == "hbm":
            peak, punit, achieved = peaks["hbm"], "GB/s", dom["units"] / (dom["ms"] * 1e-3) / 1e9
        elif dom["bound"] == "tensor":
            peak, punit, achieved = peaks["bf16_sust"], "TFLOP/s", dom["units"] / (dom["ms"] * 1e-3) / 1e12
        elif dom["bound"] == "tf32":
            peak, punit, achieved = load_tf32_peak()[0], "TFLOP/s", dom["units"] / (dom["ms"] * 1e-3) / 1e12
        else:  # fp32 FFMA on CUDA cores: 152 SMs x 128 lanes x 2 flop x max SM clock
            peak = 152 * 128 * 2 * peaks["sm_mhz"] * 1e6 / 1e12
            punit, achieved = "TFLOP/s", dom["units"] / (dom["ms"] * 1e-3) / 1e12
        traffic = None
        tpath = os.path.join(ROOT, "profiles", "traffic.json")
        if os.path.exists(tpath):
            with open(tpath) as f:
                tj = json.load(f)
            ent = tj.get(f"{args.workload}:{prec}:{dom['name']}")
            if ent and ent.get("src_hash") == sources_hash(ent.get("sources", [])):
                traffic = ent["bytes_per_launch"]
        roofline = {"kernel": dom["name"], "bound": dom["bound"], "achieved": round(achieved, 2), "peak": peak,
                    "unit": punit, "frac": round(achieved / peak, 4), "traffic": traffic,
                    "peak_source": f"{peaks['source']} ({'sustained bf16' if dom['bound'] == 'tensor' else 'copy' if dom['bound'] == 'hbm' else 'derived'})"}
    planned, compulsory = step_bytes(w, prec, args.gate, wt)
    line = {
        "metric": METRIC, "value": round(ms_step, 4), "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms_step, 4), "higher_is_better": False, "scaling": "weak",
        "vs_baseline": None, "dtype": DTYPE_NAME[prec], "data": "synthetic",
        "config": {"workload": args.workload, "layers": w.num_layers, "rank": w.rank, "shapes_per_block":
                   [list(s) for s in w.shapes[:6]], "gate_mode": args.gate, "precision": prec,
                   "l2": "no flush: each step streams far more than the 129 MB L2",
                   "matrices_per_s": round(world * w.num_layers / (ms_step * 1e-3), 1),
                   # byte models of the step with each layer's branch as taken in the timed steps
                   "step_hbm_frac_planned_bytes": round(planned / (ms_step * 1e-3) / 1e9 / peaks["hbm"], 4),
                   "step_hbm_frac_compulsory_bytes": round(compulsory / (ms_step * 1e-3) / 1e9 / peaks["hbm"], 4),
                   "sync_rate": 1.0 if wt is None else round(sum(wt) / len(wt), 4),
                   "synced_layers_per_step": sync_per_step,
                   "parallelism": f"replicas x{world}"},
        "roofline": roofline,
        "e2e": {"value": round(e2e_ms, 4), "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": launches * args.steps,
        "cuda_graph": bool(args.graph),
        "clocks": clocks,
        "kernels": [dict(name=k["name"], ms=round(k["ms"], 4), **kernel_frac(k, peaks)) for k in kern],
        "timed_steps_with_kernel_events": nsteps_timed,
    }
    return line


# ------------------------------------------------------------------- CPU (oracle) ---

def oracle_matrix_seconds(w, layer_ids, threads):
    """Runs the oracle step on the given layers in a child process with `threads` BLAS threads;
    returns the per-layer seconds."""
    env = dict(os.environ)
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        env[k] = str(threads)
    code = ("import json,sys,time\nsys.path.insert(0,%r)\nimport oracle.curvadion as oc, workloads as wl\n"
            "w=wl.WORKLOADS[%r]\nout=[]\n"
            "for l in %r:\n"
            "    X,M,Q=wl.init_layer(w,l)\n    G=wl.gradient(w,l,1)\n"
            "    lay=oc.LayerState(X=oc.as_f64(X),M=oc.as_f64(M),Q=oc.as_f64(Q))\n    g=oc.as_f64(G)\n"
            "    t=time.perf_counter()\n    oc.curvadion_step([lay],[g],[0.0],oc.HParams(),1)\n"
            "    out.append(time.perf_counter()-t)\n"
            "print(json.dumps(out))\n") % (ROOT, w.name, list(layer_ids))
    r = subprocess.run([sys.executable, "-c", code], env=env, stdout=subprocess.PIPE, text=True, check=True)
    return json.loads(r.stdout.strip().splitlines()[-1])


def cpu_baseline(args):
    import workloads as wl

    w = wl.WORKLOADS[args.workload]
    cores = os.cpu_count() or 1
    block = list(range(min(6, w.num_layers)))
    t0 = time.perf_counter()
    secs = oracle_matrix_seconds(w, block, cores)
    wall = time.perf_counter() - t0
    per_matrix = sum(secs) / len(secs)
    return {"value": round(per_matrix * w.num_layers * 1e3, 1), "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"fp64 numpy oracle, one step of the first {len(block)} matrices (one block) of {w.name}; "
                      f"value = mean s/matrix x {w.num_layers} matrices; {wall:.1f} s wall"}


def run_reference(args, rank):
    """The oracle as the reference arm: each step runs one matrix of the first block, in rotation."""
    if rank != 0:
        return None
    import workloads as wl

    w = wl.WORKLOADS[args.workload]
    cores = os.cpu_count() or 1
    block = min(6, w.num_layers)
    ids = [i % block for i in range(args.warmup + args.steps)]
    secs = oracle_matrix_seconds(w, ids, cores)
    timed = secs[args.warmup:]
    ms = (sum(timed) / len(timed)) * w.num_layers * 1e3
    return {"impl": "reference", "metric": METRIC, "value": round(ms, 1), "unit": UNIT, "n_gpus": 1,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 1), "higher_is_better": False,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": args.workload, "layers": w.num_layers, "rank": w.rank, "gate_mode": args.gate},
            "cpu_baseline": {"value": round(ms, 1), "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": f"each step: the fp64 oracle on one matrix of the first block of {w.name} "
                                       f"(rotating over {block} shapes); value = mean s/matrix x {w.num_layers}"},
            "e2e": {"value": round(ms, 1), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def measure_tf32_peak():
    """Dense tf32 throughput of cuBLAS on this GPU, measured the way the bf16 peak is: an
    8192^3 fp32 GEMM with tf32 tensor cores allowed, best of 10 (CUDA events), 2 N^3 flops."""
    import torch

    torch.backends.cuda.matmul.allow_tf32 = True
    n = 8192
    a = torch.randn(n, n, device="cuda")
    b = torch.randn(n, n, device="cuda")
    for _ in range(3):
        a @ b
    best = math.inf
    for _ in range(10):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        a @ b
        e1.record()
        torch.cuda.synchronize()
        best = min(best, e0.elapsed_time(e1))
    return {"tf32_tflops": round(2 * n ** 3 / (best * 1e-3) / 1e12, 1), "n": n, "best_ms": round(best, 4),
            "how": "torch.matmul fp32 8192^3 with allow_tf32 (cuBLAS), best of 10, CUDA events"}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--precision", default=None, choices=list(PREC))
    ap.add_argument("--gate", default="always", choices=["always", "global", "per_layer"])
    ap.add_argument("--tau", type=float, default=0.5)
    ap.add_argument("--t0", type=int, default=1, help="index of the first (warm-up) step: gradients G_t and "
                    "the step number t start there")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--tf32-peak", action="store_true", help="print the measured cuBLAS tf32 throughput and exit")
    ap.add_argument("--graph", action="store_true", help="time steps replayed from a CUDA graph (--gate always only)")
    args = ap.parse_args()
    if args.graph and args.gate != "always":
        ap.error("--graph replays one captured step, which needs --gate always (no per-step gradients)")
    if args.tf32_peak:
        print(json.dumps(measure_tf32_peak()), flush=True)
        return
    if args.warmup < 3:  # the timing rules ask for at least 3 warm-up steps; the line reports 3
        print(f"bench.py: --warmup {args.warmup} raised to 3", file=sys.stderr)
        args.warmup = 3
    if args.precision is None:
        args.precision = os.environ.get("CURVADION_BENCH_PRECISION", "bf16")

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        line = run_reference(args, rank)
        if line is not None:
            print(json.dumps(line), flush=True)
        return
    if world > 1:
        import torch
        import torch.distributed as dist

        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    line = run_ours(args, rank, world, local_rank)
    if world > 1:
        import torch.distributed as dist

        dist.destroy_process_group()
    if line is None:
        return
    if not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(args)
    else:
        line["cpu_baseline"] = None
    print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
