#!/usr/bin/env python3
"""Benchmark of the HSA hot path on GB300 (prints one JSON line on rank 0).

Step = one pass of the prefill hot path over one batch of the long-context
workload (B=2, L=32768, S=64, Hq=32, Hkv=4, d=128, top-k=8): chunk pool ->
top-k selection -> inverse index -> forward -> backward, all through the C ABI.
The decode sub-benchmark runs hsa_decode against a resident 2^26-token memory
(64 queries x 8 heads, top-k 8). Inputs are seeded synthetic tensors generated
on the device.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl hsa|reference]

N > 1 runs under torch.distributed.run: every rank processes its own batch
(weak scaling, no data-path collective); the max time over ranks is used.
--impl reference times the CPU oracle on the same workload and metric.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402

METRIC = "HSA fwd+bwd tokens/s (L=32K,S=64,k=8); decode q/s @64M memory; % roofline"
UNIT = "tokens/s"
PREFILL = synth.WORKLOADS[3]
DECODE = synth.WORKLOADS[5]


def rank_shard(w, rank):
    """The batch rank `rank` processes: the same shapes, its own seeds (rank 0 keeps the workload's), so
    that N ranks process N distinct batches with no exchange (weak scaling)."""
    return w if rank == 0 else w.with_(number=w.number + 100 * rank)


def reduce_max(x, world, device):
    """The largest of the ranks' values (every rank gets it); the step time a job reports."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist

    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def select_workload(number, batch):
    """The timed prefill workload (default: the long-context one); smaller ones serve profiling."""
    global PREFILL
    w = synth.WORKLOADS[number]
    if w.decode or not w.backward:
        raise SystemExit(f"workload {number} is not a fwd+bwd prefill workload")
    PREFILL = w.with_(B=batch) if batch else w

# dram__bytes_read.sum + dram__bytes_write.sum per launch of the dominant
# kernel from one ncu capture, keyed by the source file it was compiled from
# and that file's sha256 at capture time (reported as null once the source
# has changed).
NCU_TRAFFIC = {
    # bwd_delta + bwd_chunk + bwd_dq_merge at the long-context workload (B=2, L=32768), one launch each
    "hsa_backward": {"bytes_per_launch": 14943344128, "source": "paper_2504_16795_gb300/csrc/bwd.cu",
                     "sha256": "28d6ae98ffff41ba1617c22c33058753d7313dcaa4fd65c52aa6c661a4481473"},
}


PEAK_NOTE = "bf16 burst: the timed region lasts well under a second"


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            j = json.load(f)
        return dict(hbm=float(j["hbm_gbs"]), bf16=float(j["bf16_tflops"]),
                    bf16_sus=float(j.get("bf16_tflops_sustained", j["bf16_tflops"])), source="measured")
    except (OSError, KeyError, ValueError):
        return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, source="fallback")


def source_sha(rel):
    import hashlib

    with open(os.path.join(ROOT, rel), "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()


# ----------------------------------------------------------------------------- algorithmic work

def slot_heads(w):
    """Number of (token, query head, selected chunk) triples."""
    t = np.arange(w.L)
    keff = np.minimum(w.topk, np.minimum(t // w.S, w.Nc))
    return int(keff.sum()) * w.Hq * w.B


def visible_pairs(w):
    t = np.arange(w.L)
    return int(np.minimum(t // w.S, w.Nc).sum()) * w.B * w.Hkv


def work_model(w):
    """Algorithmic FLOPs and compulsory HBM bytes per call (one batch)."""
    bf, f4 = 2, 4
    q = w.B * w.L * w.Hq * w.d
    kv = w.B * w.L * w.Hkv * w.d
    kb = w.B * w.Nc * w.Hkv * w.d
    sel = w.B * w.L * w.Hkv * w.topk
    u = slot_heads(w)
    return {
        "hsa_chunk_pool": dict(flops=kv, bytes=kv * bf + kb * (f4 + bf)),
        "hsa_select_topk": dict(flops=2 * w.d * visible_pairs(w) + q, bytes=q * bf + kb * f4 + sel * (4 + f4)),
        "hsa_build_index": dict(flops=0, bytes=sel * 4 * 3 + w.B * w.Hkv * w.Nc * 4),
        # gathered: the K and V rows of every selected chunk, once per (t, g, j) (the token-major loads of
        # Algorithm 1); the backward gathers them again with dO and the partial gradients, about twice
        "hsa_forward": dict(flops=4 * w.S * w.d * u, bytes=q * bf * 2 + 2 * kv * bf + sel * (4 + f4 + f4),
                            gathered=sel * 2 * w.S * w.d * bf),
        "hsa_backward": dict(flops=10 * w.S * w.d * u,
                             bytes=3 * q * bf + 2 * kv * bf + kb * f4 + q * f4 + 2 * kv * f4 + sel * (4 + f4),
                             gathered=2 * sel * 2 * w.S * w.d * bf),
    }


def bound_of(flops, nbytes, pk):
    # every timed region here lasts well under a second (a few hundred ms of
    # back-to-back steps), so the tensor roofline is the burst bf16 figure
    t_tensor = flops / (pk["bf16"] * 1e12)
    t_hbm = nbytes / (pk["hbm"] * 1e9)
    return ("tensor", t_tensor) if t_tensor >= t_hbm else ("hbm", t_hbm)


# ----------------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi samples (every 100 ms) while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(prefix="clocks", suffix=".csv")
        os.close(fd)
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        self.f.close()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        try:
            rows = open(self.path).read().strip().splitlines()
        except OSError:
            rows = []
        for r in rows:
            parts = [p.strip() for p in r.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        os.unlink(self.path)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        loaded = [s for s in sm if s >= 0.5 * max(sm)] or sm
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ----------------------------------------------------------------------------- GPU arm

def run_gpu(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist

    import paper_2504_16795_gb300 as hsa

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    if not os.path.exists(hsa.lib_path()):
        if rank == 0:
            hsa.build()
        if world > 1:
            dist.barrier()
    hsa.load()
    pk = peaks()
    w = rank_shard(PREFILL, rank)
    shape = hsa.Shape(B=w.B, L=w.L, Hq=w.Hq, Hkv=w.Hkv, d=w.d, S=w.S, topk=w.topk)
    log(f"[rank {rank}] generating inputs for {w.name}")
    X = {n: synth.device_tensor(w, n, dev) for n in ("q", "K", "V", "dO")}
    wss = hsa.Workspaces(shape, dev)
    f32, i32, bf = torch.float32, torch.int32, torch.bfloat16
    sel = (w.B, w.L, w.Hkv, w.topk)
    Y = dict(kbar32=torch.empty((w.B, w.Nc, w.Hkv, w.d), dtype=f32, device=dev),
             kbar16=torch.empty((w.B, w.Nc, w.Hkv, w.d), dtype=bf, device=dev),
             idx=torch.empty(sel, dtype=i32, device=dev), s_sel=torch.empty(sel, dtype=f32, device=dev),
             offsets=torch.empty(w.B * w.Hkv * w.Nc + 1, dtype=i32, device=dev),
             entries=torch.empty(w.B * w.L * w.Hkv * w.topk, dtype=i32, device=dev),
             O=torch.empty_like(X["q"]), w=torch.empty(sel, dtype=f32, device=dev),
             dq=torch.empty(X["q"].shape, dtype=f32, device=dev),
             dK=torch.empty(X["K"].shape, dtype=f32, device=dev),
             dV=torch.empty(X["V"].shape, dtype=f32, device=dev))
    calls = ["hsa_chunk_pool", "hsa_select_topk", "hsa_build_index", "hsa_forward", "hsa_backward"]

    def step(ev=None, X=X, Y=Y):
        def mark(i):
            if ev is not None:
                ev[i].record()
        mark(0)
        hsa.chunk_pool(shape, X["K"], Y["kbar32"], Y["kbar16"])
        mark(1)
        hsa.select_topk(shape, X["q"], Y["kbar32"], Y["idx"], Y["s_sel"], ws=wss.select)
        mark(2)
        hsa.build_index(shape, Y["idx"], Y["offsets"], Y["entries"], ws=wss.index)
        mark(3)
        hsa.forward(shape, X["q"], X["K"], X["V"], Y["idx"], Y["s_sel"], Y["offsets"], Y["entries"], Y["O"],
                    Y["w"], ws=wss.forward)
        mark(4)
        hsa.backward(shape, X["q"], X["K"], X["V"], Y["kbar32"], Y["idx"], Y["w"], Y["O"], X["dO"], Y["offsets"],
                     Y["entries"], Y["dq"], Y["dK"], Y["dV"], ws=wss.backward)
        mark(5)

    def barrier():
        torch.cuda.synchronize(dev)
        if world > 1:
            dist.barrier()

    def max_over_ranks(x):
        return reduce_max(x, world, dev)

    for _ in range(args.warmup):
        step()
    barrier()
    K = args.steps
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(6)] for _ in range(K)]
    launches0 = hsa.kernel_launches()
    with ClockSampler(local_rank) as clk:
        barrier()
        wall0 = time.perf_counter()
        for i in range(K):
            step(evs[i])
        barrier()
        wall = time.perf_counter() - wall0
    launches = hsa.kernel_launches() - launches0
    clocks = clk.summary()
    ms_total = sum(evs[i][0].elapsed_time(evs[i][5]) for i in range(K))
    per_call = {c: statistics.mean(evs[i][j].elapsed_time(evs[i][j + 1]) for i in range(K))
                for j, c in enumerate(calls)}
    ms_total = max_over_ranks(ms_total)
    ms_step = ms_total / K
    tokens = w.B * w.L
    value = world * tokens * K / (ms_total / 1e3)
    log(f"[rank {rank}] {ms_step:.3f} ms/step, wall {wall / K * 1e3:.3f} ms/step, per call (ms): "
        + ", ".join(f"{c} {v:.3f}" for c, v in per_call.items()))

    # roofline per call; the dominant call is the headline
    model = work_model(w)
    kernels = {}
    for c in calls:
        m = model[c]
        bound, t_min = bound_of(m["flops"], m["bytes"], pk)
        sec = per_call[c] / 1e3
        if bound == "tensor":
            ach, peak, unit = m["flops"] / sec / 1e12, pk["bf16"], "TFLOP/s"
        else:
            ach, peak, unit = m["bytes"] / sec / 1e9, pk["hbm"], "GB/s"
        kernels[c] = {"ms": round(per_call[c], 4), "bound": bound, "achieved": round(ach, 2), "peak": peak,
                      "unit": unit, "frac": round(ach / peak, 4), "algorithmic_flops": m["flops"],
                      "algorithmic_bytes": m["bytes"], "roofline_ms": round(t_min * 1e3, 4)}
        if "gathered" in m:  # the gather reading: chunk rows delivered per second (reuse makes it exceed HBM)
            kernels[c]["gathered_bytes"] = m["gathered"]
            kernels[c]["gathered_gbs"] = round(m["gathered"] / sec / 1e9, 1)
    dom = max(calls, key=lambda c: per_call[c])
    tr = NCU_TRAFFIC.get(dom)
    traffic = None
    if tr and source_sha(tr["source"]) == tr["sha256"]:
        traffic = tr["bytes_per_launch"]
    roof = {k: kernels[dom][k] for k in ("bound", "achieved", "peak", "unit", "frac")}
    roof.update({"kernel": dom, "traffic": traffic,
                 "peak_source": f"{pk['source']} ({PEAK_NOTE if roof['bound'] == 'tensor' else 'hbm copy'})"})

    variants = None if args.no_variants else run_variants(args, dev, pk, hsa, w, X, Y, barrier, model)
    small = None if args.no_variants else run_small_configs(args, dev, pk, hsa)

    # end to end through host buffers: H2D inputs, the path, D2H outputs, every step
    e2e = None
    if not args.no_e2e:
        host_in = {n: torch.empty(X[n].shape, dtype=X[n].dtype, pin_memory=True) for n in ("q", "K", "V", "dO")}
        for n in host_in:
            host_in[n].copy_(X[n])
        host_out = {n: torch.empty(Y[n].shape, dtype=Y[n].dtype, pin_memory=True) for n in ("O", "dq", "dK", "dV")}
        h2d = sum(t.numel() * t.element_size() for t in host_in.values())
        d2h = sum(t.numel() * t.element_size() for t in host_out.values())

        # three sets of device inputs and outputs: the inputs of the next steps go up on one copy stream
        # and the outputs of earlier steps come down on another while the compute stream runs the
        # current step (the link, not the step, sets the pace, so the copies keep it busy throughout)
        n_sets = 3
        sets = [(X, Y)] + [({n: torch.empty_like(X[n]) for n in host_in},
                            dict(Y, **{n: torch.empty_like(Y[n]) for n in host_out})) for _ in range(n_sets - 1)]
        main = torch.cuda.current_stream(dev)
        up, down = torch.cuda.Stream(dev), torch.cuda.Stream(dev)

        def e2e_run(n):
            comp_done, out_done = [None] * n_sets, [None] * n_sets
            up.wait_stream(main)
            down.wait_stream(main)
            for i in range(n):
                b = i % n_sets
                Xb, Yb = sets[b]
                with torch.cuda.stream(up):
                    if comp_done[b] is not None:
                        up.wait_event(comp_done[b])  # step i - n_sets no longer reads these inputs
                    for nm, t in host_in.items():
                        Xb[nm].copy_(t, non_blocking=True)
                    ready = torch.cuda.Event()
                    ready.record(up)
                main.wait_event(ready)
                if out_done[b] is not None:
                    main.wait_event(out_done[b])  # the outputs of step i - n_sets have left
                step(None, Xb, Yb)
                comp_done[b] = torch.cuda.Event()
                comp_done[b].record(main)
                with torch.cuda.stream(down):
                    down.wait_event(comp_done[b])
                    for nm, t in host_out.items():
                        t.copy_(Yb[nm], non_blocking=True)
                    out_done[b] = torch.cuda.Event()
                    out_done[b].record(down)
            main.wait_stream(up)
            main.wait_stream(down)

        e2e_run(max(2, min(args.warmup, 4)))
        barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        e2e_run(K)
        e1.record()
        barrier()
        ms_e2e = max_over_ranks(e0.elapsed_time(e1))
        # the link alone: each direction's copies of one step, timed by themselves
        e0.record()
        for nm, t in host_in.items():
            X[nm].copy_(t, non_blocking=True)
        e1.record()
        barrier()
        h2d_ms = e0.elapsed_time(e1)
        e0.record()
        for nm, t in host_out.items():
            t.copy_(Y[nm], non_blocking=True)
        e1.record()
        barrier()
        d2h_ms = e0.elapsed_time(e1)
        e2e = {"value": world * tokens * K / (ms_e2e / 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": ms_e2e / K,
               "h2d_gbs": round(h2d / (h2d_ms / 1e3) / 1e9, 1), "d2h_gbs": round(d2h / (d2h_ms / 1e3) / 1e9, 1),
               "overlap": "three buffer sets: inputs of later steps up and outputs of earlier steps down on two copy streams while step i runs"}
        del host_in, host_out, sets

    del X, Y, wss
    torch.cuda.empty_cache()

    decode = None
    if not args.no_decode:
        decode = run_decode(args, dev, world, pk, barrier, max_over_ranks, hsa)
        decode["append"] = run_memory_append(args, dev, pk, barrier, max_over_ranks, hsa)

    prefill_1m = None
    if not args.no_prefill_1m:
        prefill_1m = run_prefill_1m(args, dev, pk, hsa, barrier, max_over_ranks)

    return dict(value=value, ms_step=ms_step, kernels=kernels, roofline=roof, e2e=e2e, clocks=clocks,
                launches=launches, decode=decode, wall_ms_step=wall / K * 1e3, variants=variants, small=small,
                prefill_1m=prefill_1m)


def run_variants(args, dev, pk, hsa, w, X, Y, barrier, model):
    """Forward and backward of the paper-default variants, and the split backward of layers sharing one
    selection, on the same inputs and selection (outside the headline's timed region)."""
    import torch

    def timed(fn, n):
        for _ in range(2):
            fn()
        barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(n):
            fn()
        e1.record()
        barrier()
        return e0.elapsed_time(e1) / n

    def frac(call, ms):
        return round(model[call]["flops"] / (ms / 1e3) / 1e12 / pk["bf16"], 4)

    n = max(args.steps, 5)
    out = {}
    for label, inner, weights in (("softmax-off-by-one", "softmax1", "softmax"), ("stick-breaking", "softmax", "stick")):
        sh = hsa.Shape(B=w.B, L=w.L, Hq=w.Hq, Hkv=w.Hkv, d=w.d, S=w.S, topk=w.topk, inner=inner, weights=weights)
        wsf = torch.empty(hsa.workspace_size(hsa.HSA_OP_FORWARD, sh), dtype=torch.uint8, device=dev)
        wsb = torch.empty(hsa.workspace_size(hsa.HSA_OP_BACKWARD, sh), dtype=torch.uint8, device=dev)

        def fwd():
            hsa.forward(sh, X["q"], X["K"], X["V"], Y["idx"], Y["s_sel"], Y["offsets"], Y["entries"], Y["O"], Y["w"],
                        ws=wsf)

        def bwd():
            hsa.backward(sh, X["q"], X["K"], X["V"], Y["kbar32"], Y["idx"], Y["w"], Y["O"], X["dO"], Y["offsets"],
                         Y["entries"], Y["dq"], Y["dK"], Y["dV"], ws=wsb)

        tf, tb = timed(fwd, n), timed(bwd, n)
        out[label] = {"hsa_forward_ms": round(tf, 4), "hsa_backward_ms": round(tb, 4),
                      "forward_frac": frac("hsa_forward", tf), "backward_frac": frac("hsa_backward", tb)}
        del wsf, wsb
    # layers sharing one selection: per layer the attention-only backward, then the selection chain once
    sh = hsa.Shape(B=w.B, L=w.L, Hq=w.Hq, Hkv=w.Hkv, d=w.d, S=w.S, topk=w.topk)
    wsa = torch.empty(hsa.workspace_size(hsa.HSA_OP_BACKWARD_ATTENTION, sh), dtype=torch.uint8, device=dev)
    wss = torch.empty(hsa.workspace_size(hsa.HSA_OP_SELECT_BACKWARD, sh), dtype=torch.uint8, device=dev)
    ds = torch.zeros(Y["idx"].shape, dtype=torch.float32, device=dev)
    dq_sel, dK_sel = torch.empty_like(Y["dq"]), torch.empty_like(Y["dK"])
    ta = timed(lambda: hsa.backward_attention(sh, X["q"], X["K"], X["V"], Y["idx"], Y["w"], X["dO"], Y["offsets"],
                                              Y["entries"], ds, Y["dq"], Y["dK"], Y["dV"], ws=wsa), n)
    ts = timed(lambda: hsa.select_backward(sh, X["q"], Y["kbar32"], Y["idx"], ds, Y["offsets"], Y["entries"], dq_sel,
                                           dK_sel, ws=wss), n)
    out["shared selection"] = {"hsa_backward_attention_ms": round(ta, 4), "hsa_select_backward_ms": round(ts, 4),
                               "attention_frac": frac("hsa_backward", ta)}
    del wsa, wss, ds, dq_sel, dK_sel
    return out


def run_decode(args, dev, world, pk, barrier, max_over_ranks, hsa):
    import torch

    w = rank_shard(DECODE, getattr(args, "rank", 0))
    if getattr(args, "decode_tokens", None):  # a smaller memory (profiling captures)
        w = w.with_(L=args.decode_tokens)
    T, Nc = w.L, w.Nc
    log(f"generating the {T}-token decode memory")
    Kmem = synth.device_tensor(w, "K", dev)
    Vmem = synth.device_tensor(w, "V", dev)
    q = synth.device_tensor(w, "q", dev)
    pshape = hsa.Shape(B=1, L=T, Hq=w.Hq, Hkv=w.Hkv, d=w.d, topk=w.topk)
    kbar32 = torch.empty((1, Nc, w.Hkv, w.d), dtype=torch.float32, device=dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    hsa.chunk_pool(pshape, Kmem.view(1, T, w.Hkv, w.d), kbar32, None, want_bf16=False)
    e1.record()
    barrier()
    pool_ms = e0.elapsed_time(e1)
    dshape = hsa.DecodeShape(Bq=w.Bq, Hq=w.Hq, Hkv=w.Hkv, d=w.d, n_chunks=Nc, topk=w.topk)
    kb = kbar32.view(Nc, w.Hkv, w.d)
    O = torch.empty_like(q)
    out = (w.Bq, w.Hkv, w.topk)
    idx = torch.empty(out, dtype=torch.int32, device=dev)
    s_sel = torch.empty(out, dtype=torch.float32, device=dev)
    wts = torch.empty(out, dtype=torch.float32, device=dev)
    # the memory index (bf16 summaries and norms) is built once per memory, like the pooling
    e0.record()
    index = hsa.decode_index(dshape, kb)
    e1.record()
    barrier()
    index_ms = e0.elapsed_time(e1)
    nws = hsa.load().hsa_decode_indexed_workspace_size(__import__("ctypes").byref(dshape.c()))
    ws = torch.empty(int(nws), dtype=torch.uint8, device=dev)
    for _ in range(args.warmup):
        hsa.decode_indexed(dshape, q, Kmem, Vmem, kb, index, O, idx, s_sel, wts, ws)
    barrier()
    steps = max(args.steps, 10)
    e0.record()
    for _ in range(steps):
        hsa.decode_indexed(dshape, q, Kmem, Vmem, kb, index, O, idx, s_sel, wts, ws)
    e1.record()
    barrier()
    ms = max_over_ranks(e0.elapsed_time(e1)) / steps
    needles = synth.needle_chunk_ids(w)
    got = idx.cpu().numpy()
    found = int(sum(int(needles[b]) in got[b, 0] for b in range(w.Bq)))
    host = None
    if not args.no_host_memory:
        ref = [t.clone() for t in (O, idx, s_sel, wts)]
        call = (lambda Kx, Vx: hsa.decode_indexed(dshape, q, Kx, Vx, kb, index, O, idx, s_sel, wts, ws))
        host = run_decode_host_memory(args, w, Kmem, Vmem, call, ref, ms, barrier, max_over_ranks)
    scan_bytes = Nc * w.Hkv * w.d * 2  # one pass over the bf16 chunk summaries
    gather_bytes = w.Bq * w.Hkv * w.topk * 2 * w.S * w.d * 2
    nbytes = scan_bytes + gather_bytes + 2 * w.Bq * w.Hq * w.d * 2
    flops = 2 * w.Bq * w.Hkv * Nc * w.d
    achieved = nbytes / (ms / 1e3) / 1e9
    del Kmem, Vmem
    torch.cuda.empty_cache()
    return {"value": world * w.Bq / (ms / 1e3), "unit": "queries/s", "ms_per_call": ms,
            "memory_tokens": T, "chunks": Nc, "queries": w.Bq, "Hq": w.Hq, "Hkv": w.Hkv, "d": w.d, "topk": w.topk,
            "needles_found": f"{found}/{w.Bq}", "pool_ms_once": pool_ms, "index_ms_once": index_ms,
            "host_memory": host,
            "path": "hsa_decode_indexed (tensor-core scan of the bf16 summaries, exact fp32 rescoring)",
            "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": pk["hbm"], "unit": "GB/s",
                         "frac": round(achieved / pk["hbm"], 4), "algorithmic_bytes": nbytes,
                         "scan": "bf16 chunk summaries", "flops": flops}}


def run_memory_append(args, dev, pk, barrier, max_over_ranks, hsa):
    """Growing a decode memory: a 2^20-token prefill appended at once (rows stored, 2^14 chunks pooled and
    indexed in one pass over the new rows), then tokens appended one by one as a decoder emits them."""
    import torch

    w = DECODE
    T, Hkv, d = 1 << 20, w.Hkv, w.d
    cap = T // w.S + 1
    wk = w.with_(L=T)
    Kn = synth.device_tensor(wk, "K", dev)
    Vn = synth.device_tensor(wk, "V", dev)
    Km = torch.empty((cap * w.S, Hkv, d), dtype=torch.bfloat16, device=dev)
    Vm = torch.empty_like(Km)
    kb = torch.zeros((cap, Hkv, d), dtype=torch.float32, device=dev)
    shape = hsa.DecodeShape(Bq=1, Hq=w.Hq, Hkv=Hkv, d=d, n_chunks=0, topk=w.topk, capacity_chunks=cap)
    index = hsa.decode_index(shape, kb)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def timed(fn, n):
        for _ in range(args.warmup):
            fn()
        barrier()
        e0.record()
        for _ in range(n):
            fn()
        e1.record()
        barrier()
        return max_over_ranks(e0.elapsed_time(e1)) / n

    # the same rows rewritten each time: the result is the same memory
    bulk_ms = timed(lambda: hsa.memory_append(shape, 0, Kn, Vn, Km, Vm, kb, index), max(args.steps, 10))
    one_k, one_v = Kn[:w.S], Vn[:w.S]

    def stream():  # the S tokens of the next chunk, one call per token
        for t in range(w.S):
            hsa.memory_append(shape, T + t, one_k[t:t + 1], one_v[t:t + 1], Km, Vm, kb, index)

    token_ms = timed(stream, 5) / w.S  # eager: one host call per token (argument checks included)
    # a serving loop replays its per-token launches from a CUDA graph
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, capture_error_mode="relaxed"):
        stream()
    token_graph_ms = timed(graph.replay, 5) / w.S
    torch.cuda.synchronize()
    kb_once = torch.empty((1, T // w.S, Hkv, d), dtype=torch.float32, device=dev)
    hsa.chunk_pool(hsa.Shape(B=1, L=T, Hq=w.Hq, Hkv=Hkv, d=d, topk=w.topk), Kn.view(1, T, Hkv, d), kb_once, None,
                   want_bf16=False)
    identical = bool(torch.equal(kb[:T // w.S], kb_once[0])) and bool(torch.equal(Km[:T], Kn))
    tok_bytes = Hkv * d * 2
    nbytes = 4 * T * tok_bytes + (T // w.S) * Hkv * d * (4 + 4 + 2) + (T // w.S) * Hkv * 4
    achieved = nbytes / (bulk_ms / 1e3) / 1e9
    del Kn, Vn, Km, Vm, kb, index, kb_once, graph
    torch.cuda.empty_cache()
    return {"prefill_tokens": T, "prefill_append_ms": round(bulk_ms, 4),
            "prefill_tokens_per_s": T / (bulk_ms / 1e3), "token_append_us": round(token_ms * 1e3, 2),
            "token_append_us_graph": round(token_graph_ms * 1e3, 2),
            "summaries_identical_to_chunk_pool": identical,
            "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": pk["hbm"], "unit": "GB/s",
                         "frac": round(achieved / pk["hbm"], 4), "algorithmic_bytes": nbytes,
                         "counted": "read K_new, V_new; write K_mem, V_mem, K̄ fp32; index: read K̄, write bf16 "
                                    "rows and norms"}}


def run_small_configs(args, dev, pk, hsa):
    """The smaller workloads, timed the same way (one step = pool, select, index, forward, backward):
    the tiny one is bound by launch latency, not by the hardware."""
    import torch

    out = {}
    for number in (1, 2):
        w = synth.WORKLOADS[number]
        shape = hsa.Shape(B=w.B, L=w.L, Hq=w.Hq, Hkv=w.Hkv, d=w.d, S=w.S, topk=w.topk)
        X = {n: synth.device_tensor(w, n, dev) for n in ("q", "K", "V", "dO")}
        wss = hsa.Workspaces(shape, dev)

        def step():
            fwd = hsa.hsa_forward_path(shape, X["q"], X["K"], X["V"], wss)
            hsa.hsa_backward_path(shape, X["q"], X["K"], X["V"], fwd, X["dO"], wss)

        for _ in range(max(args.warmup, 3)):
            step()
        torch.cuda.synchronize()
        n = 20
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(n):
            step()
        e1.record()
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / n
        model = work_model(w)
        t_min = sum(bound_of(m["flops"], m["bytes"], pk)[1] for m in model.values())
        out[w.name] = {"ms_per_step": round(ms, 4), "tokens_per_s": w.B * w.L / (ms / 1e3),
                       "roofline_ms": round(t_min * 1e3, 4), "frac": round(t_min * 1e3 / ms, 4),
                       "bound": "launch latency" if t_min * 1e3 < 0.01 * ms else "hbm/tensor",
                       "shape": f"B={w.B} L={w.L} Hq={w.Hq} Hkv={w.Hkv} d={w.d} k={w.topk}"}
        del X, wss
    torch.cuda.empty_cache()
    return out


def needle_recall(w, idx):
    """Needle queries of the 2^20-token workload: a needle query selects only needle chunks when at least k
    of them are visible, else every visible one. Returns (queries meeting it, needle queries)."""
    needles = np.sort(synth.needle_chunk_ids(w))
    toks = synth.needle_query_tokens(w)
    is_needle = np.zeros(w.Nc + 1, bool)
    is_needle[needles] = True
    nvis = np.searchsorted(needles, toks // w.S)
    sel = idx[toks]
    picked = np.where(sel >= 0, is_needle[np.clip(sel, 0, None)], False).sum(axis=1)
    return int((picked == np.minimum(nvis, w.topk)).sum()), int(toks.size)


def run_prefill_1m(args, dev, pk, hsa, barrier, max_over_ranks):
    """The 2^20-token prefill (forward only: pool -> select -> index -> forward), where selection is the
    quadratic, tensor-bound step. Per-call CUDA events on the launching stream; per-call rooflines."""
    import torch

    w = rank_shard(synth.WORKLOADS[4], getattr(args, "rank", 0))
    if getattr(args, "prefill_tokens", None):  # a shorter sequence (profiling captures)
        w = w.with_(L=args.prefill_tokens)
    shape = hsa.Shape(B=w.B, L=w.L, Hq=w.Hq, Hkv=w.Hkv, d=w.d, S=w.S, topk=w.topk)
    log(f"generating the {w.L}-token prefill inputs")
    X = {n: synth.device_tensor(w, n, dev) for n in ("q", "K", "V")}
    f32, i32 = torch.float32, torch.int32
    sel = (w.B, w.L, w.Hkv, w.topk)

    def ws(op):
        n = hsa.workspace_size(op, shape)
        return torch.empty(n, dtype=torch.uint8, device=dev) if n else None

    # pooling and selection alone (profiling captures that must keep the device memory small)
    select_only = getattr(args, "select_only", False)
    wsel = ws(hsa.HSA_OP_SELECT)
    widx, wfwd = (None, None) if select_only else (ws(hsa.HSA_OP_INDEX), ws(hsa.HSA_OP_FORWARD))
    Y = dict(kbar32=torch.empty((w.B, w.Nc, w.Hkv, w.d), dtype=f32, device=dev),
             kbar16=torch.empty((w.B, w.Nc, w.Hkv, w.d), dtype=torch.bfloat16, device=dev),
             idx=torch.empty(sel, dtype=i32, device=dev), s_sel=torch.empty(sel, dtype=f32, device=dev))
    if not select_only:
        Y.update(offsets=torch.empty(w.B * w.Hkv * w.Nc + 1, dtype=i32, device=dev),
                 entries=torch.empty(w.B * w.L * w.Hkv * w.topk, dtype=i32, device=dev),
                 O=torch.empty_like(X["q"]), w=torch.empty(sel, dtype=f32, device=dev))
    calls = ["hsa_chunk_pool", "hsa_select_topk"] + ([] if select_only else ["hsa_build_index", "hsa_forward"])

    def step(ev=None):
        def mark(i):
            if ev is not None:
                ev[i].record()
        mark(0)
        hsa.chunk_pool(shape, X["K"], Y["kbar32"], Y["kbar16"])
        mark(1)
        hsa.select_topk(shape, X["q"], Y["kbar32"], Y["idx"], Y["s_sel"], ws=wsel)
        mark(2)
        if select_only:
            return
        hsa.build_index(shape, Y["idx"], Y["offsets"], Y["entries"], ws=widx)
        mark(3)
        hsa.forward(shape, X["q"], X["K"], X["V"], Y["idx"], Y["s_sel"], Y["offsets"], Y["entries"], Y["O"], Y["w"],
                    ws=wfwd)
        mark(4)

    for _ in range(max(3, min(args.warmup, 5))):
        step()
    barrier()
    K = max(3, min(args.steps, 10))
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(K)]
    with ClockSampler(dev.index or 0) as clk:
        barrier()
        for i in range(K):
            step(evs[i])
        barrier()
    clocks = clk.summary()
    ms_total = max_over_ranks(sum(evs[i][0].elapsed_time(evs[i][len(calls)]) for i in range(K)))
    per_call = {c: statistics.mean(evs[i][j].elapsed_time(evs[i][j + 1]) for i in range(K))
                for j, c in enumerate(calls)}
    ms_step = ms_total / K
    log(f"prefill-1m: {ms_step:.3f} ms/step, per call (ms): " + ", ".join(f"{c} {v:.3f}" for c, v in per_call.items()))
    model = work_model(w)
    kernels = {}
    for c in calls:
        m = model[c]
        bound, t_min = bound_of(m["flops"], m["bytes"], pk)
        sec = per_call[c] / 1e3
        if bound == "tensor":
            ach, peak, unit = m["flops"] / sec / 1e12, pk["bf16"], "TFLOP/s"
        else:
            ach, peak, unit = m["bytes"] / sec / 1e9, pk["hbm"], "GB/s"
        kernels[c] = {"ms": round(per_call[c], 4), "bound": bound, "achieved": round(ach, 2), "peak": peak,
                      "unit": unit, "frac": round(ach / peak, 4), "algorithmic_flops": m["flops"],
                      "algorithmic_bytes": m["bytes"], "roofline_ms": round(t_min * 1e3, 4)}
        if "gathered" in m:
            kernels[c]["gathered_bytes"] = m["gathered"]
            kernels[c]["gathered_gbs"] = round(m["gathered"] / sec / 1e9, 1)
            kernels[c]["gathered_frac_of_hbm"] = round(m["gathered"] / sec / 1e9 / pk["hbm"], 4)
    ok, n_needle = needle_recall(w, Y["idx"][0, :, 0].cpu().numpy())
    del X, Y, wsel, widx, wfwd
    torch.cuda.empty_cache()
    return {"workload": f"{w.name} forward only: B={w.B} L={w.L} S={w.S} Hq={w.Hq} Hkv={w.Hkv} d={w.d} k={w.topk}, "
                        f"{w.needle_chunks} needle chunks, 1/{w.needle_query_every} of the queries carry the needle",
            "steps": K, "ms_per_step": round(ms_step, 4), "value": w.B * w.L / (ms_step / 1e3), "unit": "tokens/s",
            "kernels": kernels, "needle_queries_ok": f"{ok}/{n_needle}", "clocks": clocks,
            "peak_note": PEAK_NOTE}


def mem_available_bytes():
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("MemAvailable:"):
                    return int(line.split()[1]) * 1024
    except OSError:
        pass
    return 0


def run_decode_host_memory(args, w, Kmem, Vmem, call, ref, hbm_ms, barrier, max_over_ranks):
    """The same decode with the token memory K, V in page-locked host memory, read by the
    kernels over the CPU-GPU link (only the k selected chunks per query cross it); the
    summaries and the index stay in HBM. Outputs must equal the HBM-resident run's."""
    import torch

    need = 2 * Kmem.numel() * Kmem.element_size()
    avail = mem_available_bytes()
    if avail < 2 * need:
        return {"skipped": f"host memory available {avail / 2**30:.0f} GiB < twice the {need / 2**30:.0f} GiB memory"}
    cudart = torch.cuda.cudart()
    t0 = time.perf_counter()
    Kh = torch.empty(Kmem.shape, dtype=Kmem.dtype)
    Vh = torch.empty(Vmem.shape, dtype=Vmem.dtype)
    registered = []
    try:
        for t in (Kh, Vh):
            rc = int(cudart.cudaHostRegister(t.data_ptr(), t.numel() * t.element_size(), 2))  # mapped
            if rc != 0:
                return {"skipped": f"cudaHostRegister failed ({rc})"}
            registered.append(t)
        Kh.copy_(Kmem)
        Vh.copy_(Vmem)
        torch.cuda.synchronize()
        setup_s = time.perf_counter() - t0
        for _ in range(args.warmup):
            call(Kh, Vh)
        barrier()
        steps = max(args.steps, 10)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(steps):
            call(Kh, Vh)
        e1.record()
        barrier()
        ms = max_over_ranks(e0.elapsed_time(e1)) / steps
        out = call(Kh, Vh)
        torch.cuda.synchronize()
        identical = all(torch.equal(a, b) for a, b in zip(out, ref))
    finally:
        for t in registered:
            cudart.cudaHostUnregister(t.data_ptr())
    link_bytes = w.Bq * w.Hkv * w.topk * 2 * w.S * w.d * 2  # the selected chunks' K and V rows
    return {"ms_per_call": ms, "queries_per_s": w.Bq / (ms / 1e3), "vs_hbm_resident": round(hbm_ms / ms, 3),
            "identical_to_hbm_resident": identical, "memory_bytes_in_host": need,
            "link_bytes_per_call": link_bytes, "link_gbs": round(link_bytes / (ms / 1e3) / 1e9, 1),
            "setup_s": round(setup_s, 1),
            "layout": "K, V in cudaHostRegister-mapped host memory; summaries, index, q, O in HBM"}


# ----------------------------------------------------------------------------- CPU oracle (baseline / reference arm)

def oracle_sample(T, b=0):
    """Host inputs for the last T tokens of batch b (all groups), as fp64 [1, L, ...] arrays."""
    w = PREFILL
    t0 = w.L - T
    q = np.zeros((1, w.L, w.Hq, w.d))
    dO = np.zeros((1, w.L, w.Hq, w.d))
    q[:, t0:] = synth.bf16_to_f64(synth.host_tensor(w, "q", (b, t0, 0, 0), (b + 1, w.L, w.Hq, w.d)))
    dO[:, t0:] = synth.bf16_to_f64(synth.host_tensor(w, "dO", (b, t0, 0, 0), (b + 1, w.L, w.Hq, w.d)))
    K = synth.bf16_to_f64(synth.host_tensor(w, "K", (b, 0, 0, 0), (b + 1, w.L, w.Hkv, w.d)))
    V = synth.bf16_to_f64(synth.host_tensor(w, "V", (b, 0, 0, 0), (b + 1, w.L, w.Hkv, w.d)))
    mask = np.zeros((1, w.L), np.uint8)
    mask[0, t0:] = 1
    return q, K, V, dO, mask


def oracle_step(data):
    """Time the oracle's fwd+bwd on the sampled tokens; pooling is charged pro rata."""
    import oracle

    w = PREFILL
    q, K, V, dO, mask = data
    T = int(mask.sum())
    t0 = time.perf_counter()
    kbar32 = oracle.pool(K, w.S, f32=True)
    kbar64 = oracle.pool(K, w.S)
    t_pool = time.perf_counter() - t0
    t1 = time.perf_counter()
    idx, s_sel, _ = oracle.select(q, kbar32, w.S, w.topk, f32=True, token_mask=mask)
    oracle.forward(q, K, V, idx, s_sel, w.S, token_mask=mask)
    oracle.backward(q, K, V, kbar64, idx, s_sel, dO, w.S, token_mask=mask)
    t_rest = time.perf_counter() - t1
    return t_rest + t_pool * T / w.L


def cpu_baseline(target_s=15.0):
    import oracle

    oracle.build()
    T = 128
    sec = oracle_step(oracle_sample(T))
    T2 = int(min(4096, max(T, T * target_s / max(sec, 1e-3))))
    T2 = max(64, (T2 // 64) * 64)
    sec2 = oracle_step(oracle_sample(T2))
    return {"value": T2 / sec2, "unit": UNIT, "cores": oracle.threads(), "kind": "oracle",
            "sample": (f"fwd+bwd of the last {T2} tokens of batch 0 (all 4 groups, 32 heads) of the "
                       f"B=2 L=32768 workload; selection over all visible chunks; chunk pooling charged "
                       f"pro rata; {sec2:.1f} s of CPU time")}


def cpu_baseline_prefill_1m(target_s=12.0):
    """The oracle's select + forward on a seeded sample of rows of the 2^20-token workload (the pooling of
    the whole K timed in full), extrapolated to all rows: forward-only tokens/s. Rows are independent, so
    the per-row cost scales; the sample is drawn uniformly over the sequence."""
    import oracle

    oracle.build()
    w = synth.WORKLOADS[4]
    K = synth.bf16_to_f64(synth.host_tensor(w, "K", (0, 0, 0, 0), w.dims("K")))
    V = synth.bf16_to_f64(synth.host_tensor(w, "V", (0, 0, 0, 0), w.dims("V")))
    t0 = time.perf_counter()
    kbar32 = oracle.pool(K, w.S, f32=True)
    t_pool = time.perf_counter() - t0
    q = np.zeros((1, w.L, w.Hq, w.d))  # only the sampled rows are written (and read by the oracle)
    rng = np.random.default_rng(5004)
    done = np.zeros(w.L, bool)

    def rows_sec(n):
        toks = np.sort(rng.choice(np.nonzero(~done)[0], n, replace=False))
        done[toks] = True
        for t in toks:
            q[0, t] = synth.bf16_to_f64(synth.host_tensor(w, "q", (0, t, 0, 0), (1, t + 1, w.Hq, w.d)))[0, 0]
        mask = np.zeros((1, w.L), np.uint8)
        mask[0, toks] = 1
        t1 = time.perf_counter()
        idx, s_sel, _ = oracle.select(q, kbar32, w.S, w.topk, f32=True, token_mask=mask)
        oracle.forward(q, K, V, idx, s_sel, w.S, token_mask=mask)
        return time.perf_counter() - t1

    n0 = 64
    sec0 = rows_sec(n0)
    n1 = int(min(32768, max(n0, n0 * target_s / max(sec0, 1e-3))))
    sec1 = rows_sec(n1)
    per_row = sec1 / n1
    total = t_pool + per_row * w.L
    return {"value": w.L / total, "unit": "tokens/s", "cores": oracle.threads(), "kind": "oracle",
            "sample": (f"select + forward of {n1} rows drawn uniformly from the 2^20 tokens ({sec1:.1f} s), "
                       f"extrapolated to all rows; pooling of the whole K timed in full ({t_pool:.1f} s)"),
            "extrapolated": True}


def cpu_baseline_decode(target_s=8.0):
    """The oracle's decode call (score every chunk summary, top-k, attention over the k chunks) for the 64
    queries of the decode workload, on a prefix of its memory; the scoring scales with the number of chunks,
    so its time is extrapolated to the full 2^20 chunks. As on the GPU, pooling the memory is not part of a
    call. Returns queries/s."""
    import oracle

    oracle.build()
    w = synth.WORKLOADS[5]
    T = 1 << 20
    wp = w.with_(L=T)
    K = synth.bf16_to_f64(synth.host_tensor(wp, "K", (0, 0, 0, 0), (1, T, w.Hkv, w.d)))
    V = synth.bf16_to_f64(synth.host_tensor(wp, "V", (0, 0, 0, 0), (1, T, w.Hkv, w.d)))
    kb = oracle.pool(K, w.S, f32=True)[0]
    q = synth.bf16_to_f64(synth.host_tensor(w, "q", (0, 0, 0, 0), w.dims("q")))[0]
    reps, t_sel = 0, 0.0
    while t_sel < target_s and reps < 1000:
        t0 = time.perf_counter()
        idx, s_sel, _ = oracle.decode_select(q, kb, w.topk, f32=True)
        t_sel += time.perf_counter() - t0
        reps += 1
    Ks, Vs = oracle.gather_chunks(K[0], idx, w.S), oracle.gather_chunks(V[0], idx, w.S)
    t0 = time.perf_counter()
    oracle.decode_attend(q, Ks, Vs, idx, s_sel)
    t_att = time.perf_counter() - t0
    per_call = t_sel / reps * (w.Nc / (T // w.S)) + t_att
    return {"value": w.Bq / per_call, "unit": "queries/s", "cores": oracle.threads(), "kind": "oracle",
            "sample": (f"{reps} decode scoring passes of the {w.Bq} queries over a {T}-token prefix of the memory "
                       f"({T // w.S} chunks, {t_sel:.1f} s), scaled to {w.Nc} chunks, plus one attention over "
                       f"the {w.topk} selected chunks"),
            "extrapolated": True}


def run_reference(args, rank, world):
    if rank != 0:
        return
    import oracle

    oracle.build()
    T = 128
    data = oracle_sample(T)
    for _ in range(args.warmup):
        oracle_step(data)
    times = [oracle_step(data) for _ in range(args.steps)]
    sec = sum(times)
    value = T * args.steps / sec
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec / args.steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": config_obj(),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": oracle.threads(), "kind": "oracle",
                             "sample": f"each step: fwd+bwd of the last {T} tokens of batch 0 (all groups)"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def config_obj():
    w = PREFILL
    return {"workload": f"{w.name} HSA fwd+bwd: B={w.B} L={w.L} S={w.S} Hq={w.Hq} Hkv={w.Hkv} d={w.d} k={w.topk}",
            "B": w.B, "L": w.L, "S": w.S, "Hq": w.Hq, "Hkv": w.Hkv, "d": w.d, "topk": w.topk,
            "global_batch": w.B, "seq_len": w.L, "parallelism": "replicas (one batch per GPU)",
            "l2": "inputs larger than L2 (q, dO, O 512 MiB each; no flush)",
            "decode_workload": f"{DECODE.name}: memory {DECODE.L} tokens, {DECODE.Bq} queries x Hq={DECODE.Hq}, "
                               f"Hkv={DECODE.Hkv}, d={DECODE.d}, k={DECODE.topk}"}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=40)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["hsa", "reference"], default="hsa")
    ap.add_argument("--no-decode", action="store_true")
    ap.add_argument("--no-host-memory", action="store_true",
                    help="skip the decode over a memory kept in host memory")
    ap.add_argument("--no-variants", action="store_true", help="skip the variant and shared-selection timings")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-prefill-1m", action="store_true", help="skip the 2^20-token forward-only prefill")
    ap.add_argument("--workload", type=int, default=3, help="prefill workload number (3 is the headline)")
    ap.add_argument("--batch", type=int, default=0, help="override the workload's batch (profiling)")
    ap.add_argument("--decode-tokens", type=int, default=None,
                    help="decode memory length (default: the 2^26-token workload); for profiling captures")
    ap.add_argument("--decode-only", action="store_true",
                    help="run only the decode sub-benchmark and print its object (profiling)")
    ap.add_argument("--prefill-1m-only", action="store_true",
                    help="run only the forward-only 2^20-token prefill and print its object (profiling)")
    ap.add_argument("--select-only", action="store_true",
                    help="with --prefill-1m-only: pooling and selection alone (profiling captures)")
    ap.add_argument("--prefill-tokens", type=int, default=None,
                    help="sequence length of that prefill (default 2^20); for profiling captures")
    args = ap.parse_args()
    select_workload(args.workload, args.batch)
    rank = int(os.environ.get("RANK", "0"))
    args.rank = rank
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if args.decode_only:
        import torch

        import paper_2504_16795_gb300 as hsa

        hsa.build()
        hsa.load()
        dev = torch.device("cuda", local_rank)
        torch.cuda.set_device(dev)
        d = run_decode(args, dev, 1, peaks(), torch.cuda.synchronize, lambda x: x, hsa)
        d["append"] = run_memory_append(args, dev, peaks(), torch.cuda.synchronize, lambda x: x, hsa)
        print(json.dumps({"decode": d}), flush=True)
        return
    if args.prefill_1m_only:
        import torch

        import paper_2504_16795_gb300 as hsa

        hsa.build()
        hsa.load()
        dev = torch.device("cuda", local_rank)
        torch.cuda.set_device(dev)
        p = run_prefill_1m(args, dev, peaks(), hsa, torch.cuda.synchronize, lambda x: x)
        print(json.dumps({"prefill_1m": p}), flush=True)
        return
    import torch.distributed as dist

    if world > 1:
        import torch

        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    r = run_gpu(args, rank, world, local_rank)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        log("timing the CPU oracle baseline")
        cpu = cpu_baseline()
        if r["decode"] is not None:
            log("timing the CPU oracle decode baseline")
            r["decode"]["cpu_baseline"] = cpu_baseline_decode()
        if r["prefill_1m"] is not None:
            log("timing the CPU oracle baseline of the 2^20-token prefill")
            r["prefill_1m"]["cpu_baseline"] = cpu_baseline_prefill_1m()
    if rank == 0:
        line = {"metric": METRIC, "value": r["value"], "unit": UNIT, "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": r["ms_step"], "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "bf16", "data": "synthetic", "config": config_obj(),
                "roofline": r["roofline"], "cpu_baseline": cpu, "e2e": r["e2e"], "gpu_launches": r["launches"],
                "clocks": r["clocks"], "kernels": r["kernels"], "decode": r["decode"], "variants": r["variants"], "small_configs": r["small"],
                "prefill_1m": r["prefill_1m"],
                "wall_ms_per_step": r["wall_ms_step"]}
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
