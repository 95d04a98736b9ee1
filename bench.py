"""Benchmark of the KDN token-mixer hot path on GB300.

One step = one Diagonal-KDN training forward + backward (all steps of the
chunked forward, its adjoint) over one synthetic batch shaped like a 1.3B-model
layer: B=8, H=16, T=4096, d_k=d_v=128, bfloat16 activations, float32 state.
o and the input gradients are stored in bfloat16, the dtype of their inputs.
The forward is kdn_diag_fwd_save (o, S_T, p_T and the per-chunk context of the
backward) and the backward kdn_diag_bwd_saved (every gradient from that
context); each is one kernel.  `value` is layer tokens/s (B*T per step, summed
over ranks).  The same JSON line also carries the plain inference forward of
the same shape (kdn_diag_fwd: o, S_T, p_T, no context), the decode step
(B=256, H=16, d=128, 1024 consecutive tokens in one CUDA graph) in steps/s, the
roofline of the dominant kernel (the backward sweep) and of the forward, an
end-to-end number through host buffers, and the oracle's CPU throughput on a
bounded sample.

Algorithmic bytes count every input read once and every output written once
at its stored dtype (bf16 activations in, bf16 o and gradients out) plus the
state once per sequence: 1538 B per token-head for the diagonal forward and
2820 B for its backward at d = 128.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

With --impl reference the fp64 CPU oracle is timed on a bounded sample of the
same workload on the host cores (rank 0 only).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "KDN layer fwd+bwd tokens/s at 1 GB300 and % of roofline; decode steps/s"
B, T, H, DK, DV = 8, 4096, 16, 128, 128
DEC_B, DEC_H, DEC_STEPS = 256, 16, 1024
NAMES = ("q", "k", "v", "g", "omega", "r")


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p["bf16_tflops"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, 1900.0, "fallback"


# ---------------------------------------------------------------------------
# algorithmic work (bytes that must cross HBM once; no intermediates)

def fwd_bytes(b, t, h, dk, dv, in_bytes=2, out_bytes=2, with_state=True):
    # per token-head: q, k, g, omega (dk each) + v (dv) + r read; o (dv) written
    per_tok = (4 * dk + dv + 1) * in_bytes + dv * out_bytes
    per_seq = (dk * dv * 4 + dk * 4) if with_state else 0   # S_T, p_T written
    return b * t * h * per_tok + b * h * per_seq


def bwd_bytes(b, t, h, dk, dv, in_bytes=2, out_bytes=2):
    reads = (2 * dk + dv + 2 * dk + 1 + dv) * in_bytes          # q k v g omega r dO
    writes = (2 * dk + dv + 2 * dk + 1) * out_bytes              # dq dk dv dg domega dr
    per_seq = dk * dv * 4 + dk * 4                               # dS0, dp0
    return b * t * h * (reads + writes) + b * h * per_seq


def decode_bytes(b, h, dk, dv, in_bytes=2, out_bytes=2, variant="diag"):
    # per head-step: S and p read and written (float32); q, k, v, g, omega, r read;
    # o written, counted at the activations' dtype whatever dtype stores it.  The
    # isotropic decode of the bench has one decay, one noise and one uncertainty per head.
    per_ch = dk if variant == "diag" else 1
    state = 2 * (dk * dv * 4 + per_ch * 4)
    ins = (2 * dk + dv + 2 * per_ch + 1) * in_bytes
    return b * h * (state + ins + dv * out_bytes)


# DRAM bytes per launch of each kernel at the bench workload (B=8), from one ncu
# capture (dram__bytes_read.sum + dram__bytes_write.sum) of the current build at
# B=2 (the capture-size rule), scaled by the 4x (batch, head) sequences, which
# every byte of these one-CTA-per-sequence kernels scales with; reported as
# `traffic` only for that workload.  None: not captured for the current kernel.
NCU_TRAFFIC = {"k_wy_fwd<1>": 4 * (168267008 + 316675584), "k_fused_bwd": 4 * (469453824 + 145414400),
               "k_wy_fwd<0>": None}


def chunk_flops(dk, dv, C=64):
    # App. F chunked form per token-head: two C x C products, three C x C by
    # C x d products and three d x d products (dense-counted).
    return 10 * C * max(dk, dv) + 6 * dk * dv


# ---------------------------------------------------------------------------
# clock sampling during the timed region

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
            time.sleep(0.25)
        except OSError:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for n, val in zip(names, parts[3:7]):
                if val.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------
# distributed plumbing (one process per GPU; replicas, no data exchange)

def dist_setup(n, backend="nccl"):
    """One process per GPU (replicas): rank / local rank / world from the launcher's env."""
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world != n:
        raise SystemExit(f"--gpus {n} but WORLD_SIZE={world}")
    cuda = backend == "nccl"
    if world > 1:
        import torch.distributed as dist
        if cuda:
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    elif cuda:
        torch.cuda.set_device(0)
    return rank, local, world


def barrier(world, cuda=True):
    import torch
    if cuda:
        torch.cuda.synchronize()
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    if cuda:
        torch.cuda.synchronize()


def reduce_max(x, world, device="cuda"):
    """Max of a per-rank float over all ranks (the job's time is its slowest rank's)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def step_config(world):
    """The workload both arms report: the Diagonal KDN training step on the
    1.3B-layer shape."""
    return {"workload": "Diagonal KDN fwd+bwd, 1.3B-layer shape", "B": B, "T": T, "H": H,
            "dk": DK, "dv": DV, "activations": "bf16", "outputs": "bf16", "state": "f32",
            "parallelism": f"replicas x{world}",
            "l2": "inputs larger than L2 (each activation tensor 134 MB)"}


def job_throughput(tokens_per_rank, world, ms_per_step):
    """Whole-job tokens/s: every rank's tokens over the max-over-ranks step time."""
    return tokens_per_rank * world / (ms_per_step / 1e3)


# ---------------------------------------------------------------------------
# synthetic inputs on the device (same recipe as kdn_inputs, drawn with torch)

def device_inputs(variant, b, t, h, dk, dv, seed, dtype, per_channel=True, with_grad=True):
    import torch
    gen = torch.Generator(device="cuda")
    gen.manual_seed(seed)
    f = dict(device="cuda", generator=gen, dtype=torch.float32)
    q = torch.randn(b, t, h, dk, **f)
    q = q / q.norm(dim=-1, keepdim=True)
    k = torch.randn(b, t, h, dk, **f)
    k = k / k.norm(dim=-1, keepdim=True)
    v = torch.randn(b, t, h, dv, **f)
    gshape = (b, t, h, dk) if per_channel else (b, t, h)
    g = torch.nn.functional.logsigmoid(torch.randn(gshape, **f) + 2.0)
    wshape = (b, t, h, dk) if variant == "diag" else (b, t, h)
    om = torch.nn.functional.softplus(torch.randn(wshape, **f))
    r = torch.nn.functional.softplus(torch.randn(b, t, h, **f))
    out = {n: x.to(dtype) for n, x in zip(NAMES, (q, k, v, g, om, r))}
    if with_grad:
        out["dO"] = torch.randn(b, t, h, dv, **f).to(dtype)
    return out


# ---------------------------------------------------------------------------

def run_gpu(args):
    import torch
    import paper_2609_07816_gb300 as kdn
    from paper_2609_07816_gb300 import build as kbuild

    kbuild.build()
    rank, local, world = dist_setup(args.gpus)
    hbm, tf, peak_kind = peaks()
    global B
    B = args.batch
    dt = torch.bfloat16
    ins = device_inputs("diag", B, T, H, DK, DV, seed=1000 + rank, dtype=dt)
    x = [ins[n] for n in NAMES]
    desc = kdn.make_desc(B, T, H, DK, DV, dt, out_dtype=dt)
    ws_f = kdn.alloc_workspace(desc, 0, False)
    ws_b = kdn.alloc_workspace(desc, 0, False)
    saved = torch.empty(kdn.saved_bytes(desc), dtype=torch.uint8, device="cuda")
    o = torch.empty(B, T, H, DV, dtype=dt, device="cuda")
    ST = torch.empty(B, H, DK, DV, dtype=torch.float32, device="cuda")
    pT = torch.empty(B, H, DK, dtype=torch.float32, device="cuda")
    grads = {n: torch.empty(ins[m].shape, dtype=dt, device="cuda") for n, m in
             (("dq", "q"), ("dk", "k"), ("dv", "v"), ("dg", "g"), ("domega", "omega"),
              ("dr", "r"))}
    grads["dS0"] = torch.empty(B, H, DK, DV, dtype=torch.float32, device="cuda")
    grads["dp0"] = torch.empty(B, H, DK, dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream()

    def step(ev=None):
        if ev is not None:
            ev[0].record(stream)
        kdn.kdn_diag_fwd_save(*x, o=o, ST=ST, pT=pT, saved=saved, workspace=ws_f, out_dtype=dt)
        if ev is not None:
            ev[1].record(stream)
        if not args.fwd_only:
            kdn.kdn_diag_bwd_saved(*x, saved, ins["dO"], grads=grads, workspace=ws_b, out_dtype=dt)
        if ev is not None:
            ev[2].record(stream)

    for _ in range(args.warmup):
        step()
    launches_per_step = kdn.kdn_kernel_launches(desc, 0, 3) + (
        0 if args.fwd_only else kdn.kdn_kernel_launches(desc, 0, 4))
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(world)
    with ClockSampler(local) as clk:
        start.record(stream)
        for i in range(args.steps):
            step(evs[i])
        stop.record(stream)
        torch.cuda.synchronize()
    barrier(world)
    total_ms = reduce_max(start.elapsed_time(stop), world)
    fwd_ms = statistics.mean(e[0].elapsed_time(e[1]) for e in evs)
    bwd_ms = statistics.mean(e[1].elapsed_time(e[2]) for e in evs)
    ms_step = total_ms / args.steps
    value = job_throughput(B * T, world, ms_step)

    fb = fwd_bytes(B, T, H, DK, DV)
    bb = bwd_bytes(B, T, H, DK, DV)
    # one kernel per call: k_wy_fwd<1> (forward + context), k_fused_bwd<0,1,0,0> (backward sweep)
    fwd_roof = {"bound": "hbm", "kernel": "k_wy_fwd<1> (kdn_diag_fwd_save)",
                "achieved": fb / (fwd_ms / 1e3) / 1e9, "peak": hbm, "unit": "GB/s",
                "peak_kind": peak_kind, "algorithmic_bytes": fb, "ms": fwd_ms,
                "traffic": NCU_TRAFFIC["k_wy_fwd<1>"] if B == 8 else None}
    fwd_roof["frac"] = fwd_roof["achieved"] / hbm
    bwd_roof = {"bound": "hbm", "kernel": "k_fused_bwd<0,1,0,0> (kdn_diag_bwd_saved)",
                "achieved": bb / (bwd_ms / 1e3) / 1e9, "peak": hbm, "unit": "GB/s",
                "peak_kind": peak_kind, "algorithmic_bytes": bb, "ms": bwd_ms,
                "traffic": NCU_TRAFFIC["k_fused_bwd"] if B == 8 else None}
    bwd_roof["frac"] = bwd_roof["achieved"] / hbm
    if args.fwd_only:
        roof, other = fwd_roof, None
    else:
        roof, other = (bwd_roof, fwd_roof) if bwd_ms >= fwd_ms else (fwd_roof, bwd_roof)
    # the roofline of the step against the spec peaks, max(FLOPs / 2.25 PF, bytes / 8 TB/s):
    # the bytes term binds (the forward's FLOPs take 42 us at the bench size, its bytes 102 us)
    spec_time = (fb + bb) / 8e12
    plain = run_forward_plain(kdn, torch, args, x, hbm, peak_kind) if rank == 0 else None

    dec = (run_decode(kdn, torch, hbm, args.decode_steps)
           if rank == 0 and not args.no_decode else None)
    iso = run_iso_step(kdn, torch, args, hbm) if rank == 0 and not args.no_decode else None
    e2e = run_e2e(kdn, torch, x, ins, args) if rank == 0 and not args.no_e2e else None
    lng = run_long_context(kdn, torch, args, hbm) if rank == 0 and not args.no_long else None
    lgt = (run_logit_step(kdn, torch, args, x, o, saved, grads, ws_f, ws_b, ins["dO"])
           if rank == 0 and not args.no_decode else None)
    out = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic",
        "config": step_config(world),
        "fwd_ms": fwd_ms, "bwd_ms": bwd_ms,
        "roofline": roof, "roofline_other_kernel": other,
        "spec_roofline_frac": spec_time / (ms_step / 1e3) if ms_step > 0 else None,
        "forward_plain": plain,
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clk.summary(),
        "decode": dec, "iso_step": iso, "e2e": e2e, "long_context": lng, "logit_gates": lgt,
    }
    if rank == 0 and not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(sample_heads=args.cpu_heads)
    if rank == 0:
        print(json.dumps(out))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def run_forward_plain(kdn, torch, args, x, hbm, peak_kind):
    """The inference forward of the bench shape (B=8, H=16, T=4096, d=128):
    kdn_diag_fwd writing o (bf16), S_T and p_T, without the backward context;
    tokens/s and its roofline, against the spec peak (bytes / 8 TB/s, the
    target's formula) and against the measured copy rate."""
    dt = torch.bfloat16
    desc = kdn.make_desc(B, T, H, DK, DV, dt, out_dtype=dt)
    ws = kdn.alloc_workspace(desc, 0, False)
    o = torch.empty(B, T, H, DV, dtype=dt, device="cuda")
    ST = torch.empty(B, H, DK, DV, dtype=torch.float32, device="cuda")
    pT = torch.empty(B, H, DK, dtype=torch.float32, device="cuda")

    def fwd():
        kdn.kdn_diag_fwd(*x, o=o, ST=ST, pT=pT, workspace=ws, out_dtype=dt)

    for _ in range(args.warmup):
        fwd()
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(args.steps)]
    for e0, e1 in evs:
        e0.record(stream)
        fwd()
        e1.record(stream)
    torch.cuda.synchronize()
    ms = statistics.mean(e0.elapsed_time(e1) for e0, e1 in evs)
    nb = fwd_bytes(B, T, H, DK, DV)
    flops = B * T * H * chunk_flops(DK, DV)
    spec_s = max(nb / 8e12, flops / 2.25e15)
    return {"workload": f"Diagonal KDN forward, B={B} H={H} T={T} d=128, bf16 in / bf16 o, "
                        "f32 state (kdn_diag_fwd)",
            "value": B * T / (ms / 1e3), "unit": "tokens/s", "ms": ms,
            "gpu_launches": kdn.kdn_kernel_launches(desc, 0, 0) * args.steps,
            "spec_roofline_frac": spec_s / (ms / 1e3),
            "spec_roofline_us": spec_s * 1e6,
            "roofline": {"bound": "hbm", "kernel": "k_wy_fwd<0> (kdn_diag_fwd)",
                         "achieved": nb / (ms / 1e3) / 1e9, "peak": hbm, "unit": "GB/s",
                         "peak_kind": peak_kind, "frac": nb / (ms / 1e3) / 1e9 / hbm,
                         "algorithmic_bytes": nb,
                         "traffic": NCU_TRAFFIC["k_wy_fwd<0>"] if B == 8 else None}}


def run_iso_step(kdn, torch, args, hbm):
    """The Isotropic KDN on its 750M-layer shape (B=8, H=12, T=2048, d=128, one
    decay per head): the training step kdn_iso_fwd_save + kdn_iso_bwd_saved, and
    the inference forward kdn_iso_fwd alone, tokens/s; then both again with one
    decay per channel (the paper's layer)."""
    b, t, h = 8, 2048, 12
    ins = device_inputs("iso", b, t, h, DK, DV, seed=7, dtype=torch.bfloat16, per_channel=False)
    x = [ins[n] for n in NAMES]
    bf = torch.bfloat16
    desc = kdn.make_desc(b, t, h, DK, DV, bf, decay_per_channel=0, out_dtype=bf)
    saved = torch.empty(kdn.saved_bytes(desc, 1), dtype=torch.uint8, device="cuda")
    ws = kdn.alloc_workspace(desc, 1, False)

    def step():
        kdn.kdn_iso_fwd_save(*x, saved=saved, want_state=False, workspace=ws, out_dtype=bf)
        kdn.kdn_iso_bwd_saved(*x, saved, ins["dO"], want_state_grads=False, workspace=ws,
                              out_dtype=bf)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.steps):
        step()
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / args.steps
    # the inference forward alone (o, S_T, b_T) through kdn_iso_fwd
    o = torch.empty(b, t, h, DV, dtype=bf, device="cuda")
    ST = torch.empty(b, h, DK, DV, dtype=torch.float32, device="cuda")
    bT = torch.empty(b, h, dtype=torch.float32, device="cuda")

    def fwd():
        kdn.kdn_iso_fwd(*x, o=o, ST=ST, pT=bT, workspace=ws, out_dtype=bf)

    for _ in range(args.warmup):
        fwd()
    torch.cuda.synchronize()
    e0.record()
    for _ in range(args.steps):
        fwd()
    e1.record()
    torch.cuda.synchronize()
    fms = e0.elapsed_time(e1) / args.steps
    nb = fwd_bytes(b, t, h, DK, DV) - b * t * h * (2 * DK * 2 - 2 * 2)  # one g, omega per token
    # the paper's layer: one decay per channel (alpha_t in R^dk), same shape, both calls
    pins = device_inputs("iso", b, t, h, DK, DV, seed=8, dtype=torch.bfloat16, per_channel=True)
    px = [pins[n] for n in NAMES]
    pdesc = kdn.make_desc(b, t, h, DK, DV, bf, decay_per_channel=1, out_dtype=bf)
    psaved = torch.empty(kdn.saved_bytes(pdesc, 1), dtype=torch.uint8, device="cuda")

    def pstep():
        kdn.kdn_iso_fwd_save(*px, saved=psaved, want_state=False, workspace=ws, out_dtype=bf)
        kdn.kdn_iso_bwd_saved(*px, psaved, pins["dO"], want_state_grads=False, workspace=ws,
                              out_dtype=bf)

    def pfwd():
        kdn.kdn_iso_fwd(*px, o=o, ST=ST, pT=bT, workspace=ws, out_dtype=bf)

    res_pc = {}
    for name, fn in (("step", pstep), ("forward", pfwd)):
        for _ in range(args.warmup):
            fn()
        torch.cuda.synchronize()
        e0.record()
        for _ in range(args.steps):
            fn()
        e1.record()
        torch.cuda.synchronize()
        res_pc[name + "_ms"] = e0.elapsed_time(e1) / args.steps
    nb_pc = fwd_bytes(b, t, h, DK, DV) - b * t * h * (DK * 2 - 2)  # g per channel, one omega
    del pins, px, psaved
    return {"workload": f"Isotropic KDN fwd+bwd, B={b} H={h} T={t} d=128, one decay per head",
            "value": b * t / (ms / 1e3), "unit": "tokens/s", "ms_per_step": ms,
            "gpu_launches": 2 * args.steps,
            "forward": {"value": b * t / (fms / 1e3), "unit": "tokens/s", "ms": fms,
                        "roofline": {"bound": "hbm", "achieved": nb / (fms / 1e3) / 1e9,
                                     "peak": hbm, "unit": "GB/s",
                                     "frac": nb / (fms / 1e3) / 1e9 / hbm,
                                     "algorithmic_bytes": nb}},
            "per_channel_decay": {
                "workload": f"Isotropic KDN, B={b} H={h} T={t} d=128, one decay per channel",
                "step_value": b * t / (res_pc["step_ms"] / 1e3), "step_ms": res_pc["step_ms"],
                "forward_value": b * t / (res_pc["forward_ms"] / 1e3),
                "forward_ms": res_pc["forward_ms"], "unit": "tokens/s",
                "forward_roofline_frac": nb_pc / (res_pc["forward_ms"] / 1e3) / 1e9 / hbm}}


def run_logit_step(kdn, torch, args, x, o, saved, grads, ws_f, ws_b, dO):
    """The bench step with the gates given as logits (KDN_GATES_LOGITS: sigmoid,
    softplus and r_min + softplus applied inside the kernels, logit gradients out):
    same shape, x ~ N(2, 1), y, z ~ N(0, 1)."""
    gen = torch.Generator(device="cuda")
    gen.manual_seed(5)
    lg = [t for t in x]
    for idx, mean in ((3, 2.0), (4, 0.0), (5, 0.0)):
        lg[idx] = (torch.randn(x[idx].shape, device="cuda", generator=gen) + mean).to(x[idx].dtype)
    kw = dict(gates=kdn.KDN_GATES_LOGITS, r_min=0.01, out_dtype=o.dtype)

    def step():
        kdn.kdn_diag_fwd_save(*lg, o=o, want_state=False, saved=saved, workspace=ws_f, **kw)
        kdn.kdn_diag_bwd_saved(*lg, saved, dO, grads=grads, want_state_grads=False,
                               workspace=ws_b, **kw)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.steps):
        step()
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / args.steps
    return {"workload": f"Diagonal KDN fwd+bwd with logit gates, B={B} H={H} T={T} d=128",
            "value": B * T / (ms / 1e3), "unit": "tokens/s", "ms_per_step": ms,
            "gpu_launches": 2 * args.steps}


def run_long_context(kdn, torch, args, hbm):
    """Long-context forward, B=1 H=16 T=65536 d=128 (S_0 ~ N(0, 0.02^2), p_0 ~
    U(0.5, 2)), both variants (iso: one decay per head): kdn_*_fwd with o, S_T
    and p_T, tokens/s and the HBM roofline of the whole call.  With B*H = 16 the
    call runs sequence-parallel (8 segments of 128 chunks)."""
    b, t, h = 1, 65536, 16
    res = {}
    for variant in ("diag", "iso"):
        pc = variant == "diag"
        ins = device_inputs(variant, b, t, h, DK, DV, seed=11, dtype=torch.bfloat16,
                            per_channel=pc, with_grad=False)
        x = [ins[n] for n in NAMES]
        gen = torch.Generator(device="cuda")
        gen.manual_seed(12)
        S0 = 0.02 * torch.randn(b, h, DK, DV, device="cuda", generator=gen)
        pshape = (b, h, DK) if pc else (b, h)
        p0 = 0.5 + 1.5 * torch.rand(pshape, device="cuda", generator=gen)
        desc = kdn.make_desc(b, t, h, DK, DV, torch.bfloat16, decay_per_channel=int(pc),
                             out_dtype=torch.bfloat16)
        vi = 0 if pc else 1
        ws = kdn.alloc_workspace(desc, vi)
        o = torch.empty(b, t, h, DV, dtype=torch.bfloat16, device="cuda")
        ST = torch.empty(b, h, DK, DV, dtype=torch.float32, device="cuda")
        pT = torch.empty(pshape, dtype=torch.float32, device="cuda")
        fn = kdn.kdn_diag_fwd if pc else kdn.kdn_iso_fwd

        def call():
            fn(*x, S0, p0, o=o, ST=ST, pT=pT, workspace=ws, out_dtype=torch.bfloat16)

        for _ in range(max(3, args.warmup)):
            call()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        n = max(3, args.steps)
        e0.record()
        for _ in range(n):
            call()
        e1.record()
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / n
        nb = fwd_bytes(b, t, h, DK, DV, with_state=True)
        if not pc:  # one decay and one noise value per token-head
            nb -= b * t * h * 2 * DK * 2 - b * t * h * 2 * 2
        res[variant] = {
            "workload": f"{'Diagonal' if pc else 'Isotropic'} KDN forward, B={b} H={h} T={t} "
                        f"d=128, bf16 in / bf16 o, f32 state",
            "value": b * t / (ms / 1e3), "unit": "tokens/s", "ms": ms,
            "sequence_parallel": kdn.kdn_kernel_launches(desc, vi, 0) == 5,
            "gpu_launches": kdn.kdn_kernel_launches(desc, vi, 0),
            "roofline": {"bound": "hbm", "achieved": nb / (ms / 1e3) / 1e9, "peak": hbm,
                         "unit": "GB/s", "frac": nb / (ms / 1e3) / 1e9 / hbm,
                         "algorithmic_bytes": nb},
        }
        del ins, x, o, ws
    return res


def run_decode(kdn, torch, hbm, steps=DEC_STEPS):
    """1024 consecutive decode tokens for B=256, H=16 in one CUDA graph, both variants
    (`steps` fewer for profiling runs)."""
    DEC_STEPS = steps
    res = {}
    for variant in ("diag", "iso"):
        gen = torch.Generator(device="cuda")
        gen.manual_seed(7)
        f = dict(device="cuda", generator=gen, dtype=torch.float32)
        S = torch.randn(DEC_B, DEC_H, DK, DV, **f) * 0.02
        p = (torch.rand((DEC_B, DEC_H, DK) if variant == "diag" else (DEC_B, DEC_H), **f)
             * 1.9 + 0.1)
        shape = (DEC_STEPS, DEC_B, DEC_H)
        q = torch.randn(*shape, DK, **f)
        q = (q / q.norm(dim=-1, keepdim=True)).bfloat16()
        k = torch.randn(*shape, DK, **f)
        k = (k / k.norm(dim=-1, keepdim=True)).bfloat16()
        v = torch.randn(*shape, DV, **f).bfloat16()
        g = torch.nn.functional.logsigmoid(
            torch.randn(*shape, DK, **f) + 2.0 if variant == "diag" else torch.randn(*shape, **f) + 2.0
        ).bfloat16()
        om = torch.nn.functional.softplus(
            torch.randn(*shape, DK, **f) if variant == "diag" else torch.randn(*shape, **f)).bfloat16()
        r = torch.nn.functional.softplus(torch.randn(*shape, **f)).bfloat16()
        o = torch.empty(DEC_B, DEC_H, DV, dtype=torch.float32, device="cuda")
        fn = kdn.kdn_diag_decode_step if variant == "diag" else kdn.kdn_iso_decode_step
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            for i in range(3):
                fn(q[i], k[i], v[i], g[i], om[i], r[i], S, p, o=o, stream=s)
        torch.cuda.current_stream().wait_stream(s)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            st = torch.cuda.current_stream()
            for i in range(DEC_STEPS):
                fn(q[i], k[i], v[i], g[i], om[i], r[i], S, p, o=o, stream=st)
        graph.replay()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        graph.replay()
        e1.record()
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1)
        per = ms / DEC_STEPS
        by = decode_bytes(DEC_B, DEC_H, DK, DV, variant=variant)
        res[variant] = {"steps_per_s": DEC_STEPS / (ms / 1e3), "us_per_step": per * 1e3,
                        "achieved_GBs": by / (per / 1e3) / 1e9, "frac_hbm": by / (per / 1e3) / 1e9 / hbm,
                        "gpu_launches": DEC_STEPS}
        del graph
    return {"metric": f"decode steps/s (B=256, H=16, d=128, {DEC_STEPS} steps, CUDA graph)",
            "value": res["diag"]["steps_per_s"], "unit": "steps/s", **res}


def run_e2e(kdn, torch, x, ins, args):
    """Same step through the public API with host buffers.  Every step uploads its
    inputs (q, k, v, g, omega, r, dO) from pinned host memory, runs the forward and
    backward, and reads its result back to the host: the layer's loss
    <dO, o>, whose gradients the backward computes.  The upload of step i+1 runs on
    a copy stream while step i computes (double-buffered device inputs), as a
    training input pipeline would."""
    names = NAMES + ("dO",)
    host_in = {n: ins[n].cpu().pin_memory() for n in names}
    bufs = [{n: torch.empty_like(ins[n]) for n in names} for _ in range(2)]
    comp = torch.cuda.current_stream()
    copy = torch.cuda.Stream()
    bf = torch.bfloat16
    desc = kdn.make_desc(B, T, H, DK, DV, bf, out_dtype=bf)
    saved = torch.empty(kdn.saved_bytes(desc), dtype=torch.uint8, device="cuda")
    ws = kdn.alloc_workspace(desc, 0, False)
    o = torch.empty(B, T, H, DV, dtype=bf, device="cuda")
    grads = {n: torch.empty(ins[m].shape, dtype=bf, device="cuda") for n, m in
             (("dq", "q"), ("dk", "k"), ("dv", "v"), ("dg", "g"), ("domega", "omega"),
              ("dr", "r"))}
    nmax = args.warmup + args.steps
    loss_host = torch.empty(nmax, dtype=torch.float32, pin_memory=True)
    copied = [torch.cuda.Event() for _ in range(2)]
    freed = [torch.cuda.Event() for _ in range(2)]

    def upload(i):
        b = i % 2
        copy.wait_event(freed[b])
        with torch.cuda.stream(copy):
            for n in names:
                bufs[b][n].copy_(host_in[n], non_blocking=True)
        copied[b].record(copy)

    def compute(i):
        b = i % 2
        comp.wait_event(copied[b])
        xx = [bufs[b][n] for n in NAMES]
        kdn.kdn_diag_fwd_save(*xx, o=o, want_state=False, saved=saved, workspace=ws, out_dtype=bf)
        kdn.kdn_diag_bwd_saved(*xx, saved, bufs[b]["dO"], grads=grads, want_state_grads=False,
                               workspace=ws, out_dtype=bf)
        loss = torch.sum(o.view(-1).float() * bufs[b]["dO"].view(-1).float(), dtype=torch.float32)
        freed[b].record(comp)
        loss_host[i].copy_(loss, non_blocking=True)

    def run(i0, n):
        upload(i0)
        for i in range(i0, i0 + n):
            if i + 1 < i0 + n:
                upload(i + 1)
            compute(i)

    run(0, args.warmup)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(comp)
    copy.wait_event(e0)
    run(args.warmup, args.steps)
    e1.record(comp)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / args.steps
    assert bool(torch.isfinite(loss_host[args.warmup:]).all())
    h2d = sum(t.numel() * t.element_size() for t in host_in.values())
    return {"value": B * T / (ms / 1e3), "unit": "tokens/s", "ms_per_step": ms,
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": 4,
            "result": "loss <dO, o> read back every step; upload of step i+1 overlaps step i"}


# ---------------------------------------------------------------------------
# CPU oracle timing (bounded sample of the same workload)

def cpu_baseline(sample_heads=None):
    import numpy as np

    import oracle
    from kdn_inputs import make_inputs
    oracle.build()
    cores = os.cpu_count() or 1
    n = sample_heads or B * H  # the whole workload's (batch, head) sequences, ~5 s on 16 cores
    ins = make_inputs("diag", 1, T, n, DK, DV, dtype="bf16", seed=0, with_grad=True)
    args = [ins[k] for k in NAMES]
    t0 = time.perf_counter()
    r1 = oracle.fwd("diag", *args, None, None, threads=cores)
    r2 = oracle.bwd("diag", *args, None, None, ins["dO"], threads=cores)
    wall = time.perf_counter() - t0
    token_heads = n * T
    return {"value": token_heads / H / wall, "unit": "tokens/s", "cores": int(r2["threads"]),
            "kind": "oracle", "wall_s": wall,
            "sample": f"fwd+bwd of {n} (batch, head) sequences of T={T}, d=128 "
                      f"(= {token_heads / H:.0f} layer tokens of H={H})"}


def run_reference(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import oracle
    oracle.build()
    cores = os.cpu_count() or 1
    n = B * H
    samples = []
    for i in range(args.warmup + args.steps):
        cb = cpu_baseline(sample_heads=n)
        if i >= args.warmup:
            samples.append(cb)
    val = statistics.mean(s["value"] for s in samples)
    ms = statistics.mean(s["wall_s"] for s in samples) * 1e3
    out = {"impl": "reference", "metric": METRIC, "value": val, "unit": "tokens/s",
           "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
           "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
           "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": dict(step_config(world), sample=samples[0]["sample"]),
           "cpu_baseline": {"value": val, "unit": "tokens/s", "cores": samples[0]["cores"],
                            "kind": "oracle", "sample": samples[0]["sample"]},
           "e2e": {"value": val, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="kdn", choices=["kdn", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-decode", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-long", action="store_true", help="skip the long-context forward")
    ap.add_argument("--decode-steps", type=int, default=DEC_STEPS,
                    help="decode tokens per graph (profiling runs only)")
    ap.add_argument("--fwd-only", action="store_true", help="profiling runs: forward only")
    ap.add_argument("--batch", type=int, default=B, help="batch size (profiling runs only)")
    ap.add_argument("--cpu-heads", type=int, default=None)
    args = ap.parse_args()
    if args.warmup < 3 and args.impl != "reference":
        raise SystemExit("--warmup must be >= 3")
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
