"""Benchmark of the whole-model delta -> TopKMask -> update/merge pass.

One step = one pass of the hot path over a full synthetic parameter set held
in HBM.  Default workload: the Qwen2.5-7B-shaped fused delta + mask + update
(bf16 base and RL checkpoint, 254 tensors, 7,615,483,904 parameters,
per-tensor TopKMask density 5 %, masked ISO update).  Other workloads
(--workload) are for investigation.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl mine|reference]

Prints one JSON line.  Under torchrun (N > 1) every rank runs its own copy of
the workload (weak scaling, no data-path collective); the step time is the
maximum over ranks.
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2607_19331_gb300.shard import job_throughput, reduce_step_ms  # noqa: E402

METRIC = "G params/s and achieved HBM GB/s (% of ~8 TB/s) for full-model mask+merge"
UNIT = "Gparams/s"
NOMINAL_HBM_GBS = 8000.0

WORKLOADS = {
    # name: (shape set, K, op, inputs, density, scope, description)
    "qwen1.5b_update": ("qwen1.5b", 1, "iso", "ckpt_bf16", 0.05, "tensor",
                        "Qwen2.5-1.5B-shaped bf16 base + RL checkpoint, masked ISO update, "
                        "per-tensor TopKMask 5%"),
    "qwen7b_update": ("qwen7b", 1, "iso", "ckpt_bf16", 0.05, "tensor",
                      "Qwen2.5-7B-shaped bf16 base + RL checkpoint, fused delta+mask+update, "
                      "per-tensor TopKMask 5%"),
    "qwen7b_ties_k8": ("qwen7b", 8, "ties", "delta_f32", 0.10, "tensor",
                       "Qwen2.5-7B-shaped bf16 base, 8 fp32 RL deltas, TopKMask 10% + TIES"),
    "qwen7b_iso_k8": ("qwen7b", 8, "iso", "delta_f32", 0.10, "tensor",
                      "Qwen2.5-7B-shaped bf16 base, 8 fp32 RL deltas, TopKMask 10% + ISO retention"),
    "qwen7b_update_global": ("qwen7b", 1, "ties", "ckpt_bf16", 0.20, "global",
                             "Qwen2.5-7B-shaped bf16 base + RL checkpoint, TIES update under one "
                             "GLOBAL TopKMask at 20% over the whole task vector (the paper's TIES "
                             "scope and density)"),
    "qwen7b_ram_k8": ("qwen7b", 8, "ram", "delta_f32", 0.0, "tensor",
                      "Qwen2.5-7B-shaped bf16 base, 8 fp32 RL deltas, RAM merge (eps_act 1e-5, no trim)"),
    "sweep_tensor": ("sweep", 1, "ties", "delta_bf16", 0.05, "tensor",
                     "bf16 4096x14336 delta N(0,1e-3^2)+1e-3 t_3 with 1000 threshold ties, "
                     "per-tensor TopKMask + masked update (--density)"),
    "sweep_block": ("sweep", 1, "ties", "delta_bf16", 0.05, "block",
                    "bf16 4096x14336 delta N(0,1e-3^2)+1e-3 t_3 with 1000 threshold ties, "
                    "per-128x128-block TopKMask + masked update (--density)"),
}


def fused_pass(K, inputs, op, scope, two_pass=False):
    """Whether the library runs the K = 1 update as its fused single pass
    (bf16 base and update, per-tensor TopKMask, a trimming operator)."""
    return (not two_pass and K == 1 and scope == "tensor" and op not in ("ta", "ram")
            and inputs in ("ckpt_bf16", "delta_bf16"))


def algorithmic_bytes(shapes, K, inputs, op, scope="tensor", two_pass=False):
    """Bytes each full pass must move at minimum, per kernel kind.

    apply:        read theta_0 and the K experts once, write the output once
    count:        (per-tensor scope) read the K task vectors once; in the fused
                  K = 1 pass this kernel is the whole update (read theta_0 and
                  the expert, write the output) and there is no apply pass
    block_select: (per-block scope) read the K task vectors once; for the
                  K = 1 TIES update this kernel writes the outputs itself (read
                  theta_0 and the expert, write the output) and there is no
                  apply pass
    gram:         (ISO, K >= 2) read the K task vectors once
    """
    n_all = sum(r * c for r, c, _ in shapes)
    n_trim = sum(r * c for r, c, one in shapes if not (one and op == "iso"))
    per_x = {"ckpt_bf16": 2, "delta_bf16": 2, "delta_f32": 4}[inputs]
    per_base, per_out = 2, 2
    if fused_pass(K, inputs, op, scope, two_pass):
        return {"count": n_all * (per_base + per_x + per_out)}
    if K == 1 and scope == "block" and op == "ties":
        return {"block_select": n_all * (per_base + per_x + per_out)}
    read_tau = n_trim * (K * per_x + (per_base if inputs == "ckpt_bf16" else 0))
    out = {"apply": n_all * (per_base + K * per_x + per_out)}
    if op not in ("ta", "ram"):   # the trimming operators select first
        out["block_select" if scope == "block" else "count"] = read_tau
    if op == "iso" and K >= 2:
        out["gram"] = read_tau
    return out


# the source files each timed kernel kind is built from (besides the shared headers)
KERNEL_SOURCES = {
    "count": ["iso_fused.cu", "iso_select.cu"],   # fused K = 1 pass, or the two-pass counting read
    "apply": ["iso_apply.cu", "iso_merge.cu"],
    "merge": ["iso_merge.cu"],                    # the apply pass of K >= 2 (and RAM) runs k_merge alone
    "gram": ["iso_merge.cu"],
    "block_select": ["iso_block.cu"],
}


def _code_only(text: bytes) -> bytes:
    """The source without comments and with whitespace collapsed: edits to
    comments leave a kernel's hash, and so its profiled traffic, in place."""
    import re
    t = text.decode()
    t = re.sub(r"/\*.*?\*/", " ", t, flags=re.S)
    t = re.sub(r"//[^\n]*", " ", t)
    return " ".join(t.split()).encode()


def kernel_source_hash(kind=None):
    """sha1 of a kernel kind's sources and the shared headers (all sources
    when kind is None), comments and whitespace left out: a profile's traffic
    applies only to the kernels it measured."""
    import hashlib
    csrc = os.path.join(ROOT, "paper_2607_19331_gb300", "csrc")
    names = KERNEL_SOURCES.get(kind) if kind else None
    if names is None:
        names = sorted(f for f in os.listdir(csrc) if f.endswith(".cu"))
    files = [os.path.join(csrc, f) for f in sorted(names) + ["iso_internal.cuh", "iso_kernels.cuh"]]
    files.append(os.path.join(ROOT, "include", "iso.h"))
    h = hashlib.sha1()
    for f in files:
        h.update(os.path.basename(f).encode())
        with open(f, "rb") as fh:
            h.update(_code_only(fh.read()))
    return h.hexdigest()[:16]


def profiled_traffic(kernel, workload):
    """DRAM bytes per parameter of `kernel` from the committed ncu summaries in
    profiles/, if they were taken on the kernel's current sources."""
    import glob
    sha = kernel_source_hash(kernel)
    for f in glob.glob(os.path.join(ROOT, "profiles", "*.md")):
        for line in open(f):
            if not line.startswith("traffic:"):
                continue
            kv = dict(x.split("=", 1) for x in line.split()[1:])
            if kv.get("kernel") == kernel and kv.get("workload") == workload and kv.get("csrc_sha1") == sha:
                return float(kv["dram_bytes_per_param"])
    return None


def read_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class Clocks:
    """nvidia-smi sampler for the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, path: str):
        self.path = path
        self.idx = gpu_index
        self.p = None
        try:
            self.f = open(path, "w")
            self.p = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                                       "-i", str(gpu_index), "-lms", "100"], stdout=self.f,
                                      stderr=subprocess.DEVNULL)
        except Exception:
            self.p = None

    def stop(self):
        if self.p is None:
            return None
        self.p.terminate()
        try:
            self.p.wait(timeout=5)
        except Exception:
            self.p.kill()
        self.f.close()
        rows = []
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), parts[5:9]))
            except ValueError:
                continue
        if not rows:
            return None
        sm = sorted(r[0] for r in rows)
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i, v in enumerate(r[2]) if v.lower() == "active"})
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


def make_workload(name, device, seed, layers=None, density=None, scale=1, shard=None):
    """The workload's tensors on `device`; with shard = (rank, world) only the
    tensors shard_tensors assigns to this rank (the same seeded values the
    whole set would hold)."""
    import torch
    import synth
    shapes_name, K, op, inputs, d0, scope, desc = WORKLOADS[name]
    if shapes_name == "sweep":
        shapes = [(4096, 14336, False)]
        th0 = synth.base_weights(shapes, seed=seed, device=device)
        experts = [[synth.density_sweep_delta(seed=seed, rho=d0 if density is None else density,
                                              device=device)]]
        torch.cuda.synchronize()
        return shapes, th0, experts
    shapes = synth.qwen_shapes(shapes_name, layers=layers, scale=scale)
    if inputs == "ckpt_bf16":
        th0, th1 = synth.rl_update_set(shapes, seed=seed, device=device)
        experts = [th1]
    else:
        th0 = synth.base_weights(shapes, seed=seed, device=device)
        experts, _ = synth.merge_experts(shapes, seed=seed, K=K, device=device)
    if shard is not None:
        from paper_2607_19331_gb300.shard import shard_tensors
        mine = shard_tensors([r * c for r, c, _ in shapes], shard[1])[shard[0]]
        shapes = [shapes[q] for q in mine]
        th0 = [th0[q] for q in mine]
        experts = [[e[q] for q in mine] for e in experts]
        torch.cuda.empty_cache()
    torch.cuda.synchronize()
    return shapes, th0, experts


def run_frame(args):
    """The frame-space ISO-Merger (App. E) of one Qwen2.5-7B gate/up
    projection (3584 x 18944, bf16 base ~ N(0, 0.02^2), K RL experts = base +
    N(0, (5e-4)^2), seeded).  The thin SVDs (torch.linalg, binary64, the one
    library step) are timed once and reported apart; a step is one
    iso_frame_merge call on resident factors.  The roofline is that of the
    dominant kernel, the tcgen05 product, timed live on the reconstruction's
    shape (M = 3584, N = 18944, a contraction of 3 x 2 x 3584 tf32 terms)."""
    import torch
    import paper_2607_19331_gb300 as iso
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    m, n, K = args.frame_m, args.frame_n, args.experts
    g = torch.Generator(device=dev).manual_seed(0)
    W0 = (torch.randn(m, n, generator=g, device=dev) * 0.02).to(torch.bfloat16)
    ex = [(W0.float() + torch.randn(m, n, generator=g, device=dev) * 5e-4).to(torch.bfloat16) for _ in range(K)]
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    U0, S0, Vt0 = iso.thin_svd(W0)
    fac = [iso.thin_svd(e) for e in ex]
    torch.cuda.synchronize()
    svd_s = time.perf_counter() - t0
    out = torch.empty_like(W0)
    ws = iso.Workspace(dev)
    ws.get(iso.frame_workspace_size(m, n, K))
    stream = torch.cuda.current_stream(dev)

    def step():
        iso.frame_merge_factors(U0, S0, Vt0, [f[0] for f in fac], [f[2] for f in fac], W0, out=out,
                                workspace=ws, stream=stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    clocks = Clocks(0, args.clock_log or os.path.join(__import__("tempfile").gettempdir(), "iso_clocks_frame.csv"))
    time.sleep(0.3)
    l0 = iso.launch_count()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / args.steps
    ck = clocks.stop()
    launches = (iso.launch_count() - l0) // max(1, args.steps)
    iso.profile_reset()
    iso.profile_enable(True)
    for _ in range(3):
        step()
    torch.cuda.synchronize()
    prof = iso.profile_read()
    iso.profile_enable(False)
    # the dominant kernel alone, on the reconstruction's shape
    pad = lambda x: (x + 127) // 128 * 128
    Mp, Np, L = pad(m), pad(n), 2 * pad(min(m, n))
    A = torch.randn(Mp, 4 * L, device=dev)
    B = torch.randn(Np, 4 * L, device=dev)
    C = torch.empty(Mp, Np, device=dev)
    for _ in range(3):
        iso.gemm_tf32(A, B, C, 3 * L, 0, L)
    torch.cuda.synchronize()
    f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = 10
    f0.record(stream)
    for _ in range(reps):
        iso.gemm_tf32(A, B, C, 3 * L, 0, L)
    f1.record(stream)
    torch.cuda.synchronize()
    g_ms = f0.elapsed_time(f1) / reps
    flops = 2.0 * Mp * Np * 3 * L
    achieved = flops / (g_ms * 1e-3) / 1e12
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            pk = json.load(f)
        peak, src = float(pk["bf16_tflops"]) * 1.1 / 2.25, "measured bf16 burst x nominal tf32/bf16 (1.1/2.25)"
    except Exception:
        peak, src = 1900.0 * 1.1 / 2.25, "fallback bf16 x nominal tf32/bf16 (1.1/2.25)"
    line = {
        "metric": "frame-space ISO-Merger: matrix params/s (one projection)", "value": round(m * n / (ms * 1e-3) / 1e9, 4),
        "unit": "Gparams/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms, 3), "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "tf32x3 products, f32 accumulation, f64 q x q algebra", "data": "synthetic (seeded)",
        "config": {"workload": args.workload, "m": m, "n": n, "experts": K,
                   "svd_seconds_library": round(svd_s, 2),
                   "l2": "operands larger than L2 (129 MB); no flush needed"},
        "kernels": {k: {"launches": v[0] // 3, "ms_per_step": round(v[1] / 3, 3)} for k, v in prof.items()},
        "roofline": {"bound": "tensor", "kernel": "k_gemm_tf32 (reconstruction shape)", "achieved": round(achieved, 1),
                     "peak": round(peak, 1), "peak_source": src, "unit": "TFLOP/s",
                     "frac": round(achieved / peak, 4), "traffic": None, "avg_launch_ms": round(g_ms, 3),
                     "algorithmic_flops_per_launch": flops},
        "gpu_launches": int(launches), "clocks": ck, "e2e": None, "cpu_baseline": None,
    }
    print(json.dumps(line), flush=True)


def run_opt(args):
    """One ISO[AdamW] step (Sec. 4.3) of a Qwen2.5-7B gate/up projection
    (3584 x 18944, bf16 weights, binary64 frames from the weights' thin SVD,
    a seeded synthetic gradient ~ N(0, 1e-3^2)) at the paper's learning rate
    7.5e-7.  A step is one iso_opt_step call; the roofline is that of the
    step's tcgen05 factor-gradient product (M = 18944, N = 3584, a
    contraction of 3 x 3584 tf32 terms), timed live."""
    import torch
    import paper_2607_19331_gb300 as iso
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    m, n = args.frame_m, args.frame_n
    g = torch.Generator(device=dev).manual_seed(0)
    W = (torch.randn(m, n, generator=g, device=dev) * 0.02).to(torch.bfloat16)
    G = torch.randn(m, n, generator=g, device=dev) * 1e-3
    t0 = time.perf_counter()
    U, S0, Vt = iso.thin_svd(W)
    torch.cuda.synchronize()
    svd_s = time.perf_counter() - t0
    V = Vt.t().contiguous()
    moms = [torch.zeros_like(U, dtype=torch.float32), torch.zeros_like(U, dtype=torch.float32),
            torch.zeros_like(V, dtype=torch.float32), torch.zeros_like(V, dtype=torch.float32)]
    ws = iso.Workspace(dev)
    ws.get(iso.opt_workspace_size(m, n))
    stream = torch.cuda.current_stream(dev)
    state = {"t": 0}

    def step():
        state["t"] += 1
        iso.opt_step(U, V, S0, G, *moms, W, W_out=W, lr=7.5e-7, step=state["t"], workspace=ws, stream=stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    clocks = Clocks(0, args.clock_log or os.path.join(__import__("tempfile").gettempdir(), "iso_clocks_opt.csv"))
    time.sleep(0.3)
    l0 = iso.launch_count()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / args.steps
    ck = clocks.stop()
    launches = (iso.launch_count() - l0) // max(1, args.steps)
    iso.profile_reset()
    iso.profile_enable(True)
    for _ in range(3):
        step()
    torch.cuda.synchronize()
    prof = iso.profile_read()
    iso.profile_enable(False)
    pad = lambda x: (x + 127) // 128 * 128
    Np, L = pad(n), pad(m)
    A = torch.randn(Np, 4 * L, device=dev)
    B = torch.randn(pad(min(m, n)), 4 * L, device=dev)
    C = torch.empty(Np, pad(min(m, n)), device=dev)
    for _ in range(3):
        iso.gemm_tf32(A, B, C, 3 * L, 0, L)
    torch.cuda.synchronize()
    f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    f0.record(stream)
    for _ in range(10):
        iso.gemm_tf32(A, B, C, 3 * L, 0, L)
    f1.record(stream)
    torch.cuda.synchronize()
    g_ms = f0.elapsed_time(f1) / 10
    flops = 2.0 * Np * pad(min(m, n)) * 3 * L
    achieved = flops / (g_ms * 1e-3) / 1e12
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            peak, src = float(json.load(f)["bf16_tflops"]) * 1.1 / 2.25, "measured bf16 burst x nominal tf32/bf16 (1.1/2.25)"
    except Exception:
        peak, src = 1900.0 * 1.1 / 2.25, "fallback bf16 x nominal tf32/bf16 (1.1/2.25)"
    line = {
        "metric": "ISO[AdamW] step: matrix params/s (one projection)", "value": round(m * n / (ms * 1e-3) / 1e9, 4),
        "unit": "Gparams/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "tf32x3 products, f32 accumulation, f64 frames and AdamW arithmetic", "data": "synthetic (seeded)",
        "config": {"workload": args.workload, "m": m, "n": n, "lr": 7.5e-7, "svd_seconds_library_once": round(svd_s, 2),
                   "l2": "operands larger than L2 (129 MB); no flush needed"},
        "kernels": {k: {"launches": v[0] // 3, "ms_per_step": round(v[1] / 3, 3)} for k, v in prof.items()},
        "roofline": {"bound": "tensor", "kernel": "k_gemm_tf32 (factor-gradient shape)", "achieved": round(achieved, 1),
                     "peak": round(peak, 1), "peak_source": src, "unit": "TFLOP/s", "frac": round(achieved / peak, 4),
                     "traffic": None, "avg_launch_ms": round(g_ms, 3), "algorithmic_flops_per_launch": flops},
        "gpu_launches": int(launches), "clocks": ck, "e2e": None, "cpu_baseline": None,
    }
    print(json.dumps(line), flush=True)


def run_mine(args):
    import torch
    import torch.distributed as dist
    import paper_2607_19331_gb300 as iso

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    name = args.workload
    shapes_name, K, op, inputs, density, scope, desc = WORKLOADS[name]
    if args.density is not None:
        density = args.density
    shapes, th0, experts = make_workload(name, dev, seed=0 if args.shard else rank, layers=args.layers,
                                         density=density, scale=args.scale,
                                         shard=(rank, world) if args.shard else None)
    n_params = sum(t.numel() for t in th0)
    n_params_all = n_params
    if args.shard and world > 1:
        t_n = torch.tensor([n_params], dtype=torch.int64, device=dev)
        dist.all_reduce(t_n)
        n_params_all = int(t_n.item())
    ckpt = inputs == "ckpt_bf16"
    out = [torch.empty_like(t) for t in th0]
    iso.force_two_pass(args.two_pass)
    iso.compact_candidates(args.compact_candidates)
    cfg = iso.merge_cfg(op, density, scope)
    mn, full = iso.iso_workspace_size(th0, K, cfg)
    free = torch.cuda.mem_get_info(dev)[0]
    ws_bytes = full if full + (1 << 30) < free else max(mn, free - (2 << 30))
    ws = iso.Workspace(dev)
    ws.get(ws_bytes)
    stream = torch.cuda.current_stream(dev)

    def step():
        iso.iso_merge(th0, experts, op=op, experts_are_deltas=not ckpt, out=out, density=density,
                      scope=scope, lam=1.0, workspace=ws, ws_bytes=ws_bytes, stream=stream)

    def barrier():
        if world > 1:
            dist.barrier()

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    barrier()
    clocks = None
    if rank == 0:
        import tempfile
        fd, clock_path = tempfile.mkstemp(prefix="iso_clocks_", suffix=".csv")
        os.close(fd)
        clocks = Clocks(local, args.clock_log or clock_path)
    time.sleep(0.3 if clocks else 0)
    l0 = iso.launch_count()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    barrier()
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    launches = (iso.launch_count() - l0) // max(1, args.steps)
    ms = e0.elapsed_time(e1) / args.steps
    ck = clocks.stop() if clocks else None
    ms = reduce_step_ms(ms, dev)
    n_job = n_params_all if args.shard else world * n_params
    value = job_throughput(n_job, ms)

    # per-kernel device time through the library's event brackets
    iso.profile_reset()
    iso.profile_enable(True)
    prof_steps = max(3, min(args.steps, 10))
    for _ in range(prof_steps):
        step()
    torch.cuda.synchronize()
    prof = iso.profile_read()
    iso.profile_enable(False)
    algo = algorithmic_bytes(shapes, K, inputs, op, scope, args.two_pass)
    peak, peak_src = read_peaks()
    kernels = {k: {"launches": n // prof_steps, "ms_per_step": tot / prof_steps} for k, (n, tot) in prof.items()}
    dom = max(algo, key=lambda k: prof.get(k, (0, 0.0))[1])
    n_dom, t_dom = prof.get(dom, (1, 0.0))
    avg_ms = t_dom / max(1, n_dom)
    per_launch_bytes = algo[dom] / max(1, n_dom // prof_steps)
    achieved = per_launch_bytes / (avg_ms * 1e-3) / 1e9 if avg_ms > 0 else 0.0
    step_gbs = sum(algo.values()) / (ms * 1e-3) / 1e9
    small = args.layers is not None or args.scale != 1
    # the apply pass of K >= 2 merges (and of RAM at any K) is k_merge alone:
    # its traffic is tied to that kernel's sources
    hkind = "merge" if dom == "apply" and (K >= 2 or op == "ram") else dom
    tb = profiled_traffic(hkind, name) if not small else None
    traffic = None if tb is None else int(tb * n_params)

    # end to end through the public API from page-locked host memory: the
    # library's host-staged update (copies in, update, copies out, pipelined
    # over tensor groups on three streams)
    e2e = None
    if not args.no_e2e and K == 1:
        h0 = pinned_flat(th0)
        h1 = pinned_flat(experts[0])
        del th0, experts
        out.clear()
        ws.buf = torch.empty(0, dtype=torch.uint8, device=dev)
        torch.cuda.empty_cache()
        ho = pinned_flat(h0, copy=False)
        link = link_rates(dev)
        host = iso.HostUpdate(dev, group_bytes=args.e2e_group_mb << 20)
        kw = dict(op=op, update_is_delta=not ckpt, density=density, scope=scope)
        for _ in range(3):
            host.run(h0, h1, out=ho, **kw)
        torch.cuda.synchronize()
        n_e2e = max(3, min(args.steps, 5))
        evs = [torch.cuda.Event(enable_timing=True) for _ in range(n_e2e + 1)]
        evs[0].record(stream)
        for q in range(n_e2e):
            host.run(h0, h1, out=ho, **kw)
            evs[q + 1].record(stream)
        torch.cuda.synchronize()
        per = sorted(evs[q].elapsed_time(evs[q + 1]) for q in range(n_e2e))
        ms_e2e = reduce_step_ms(evs[0].elapsed_time(evs[-1]) / n_e2e, dev)
        # the host link is shared with the rest of the machine and its rate
        # varies from one measurement to the next: measure it again after the
        # timed steps and keep the best rate seen as the link's capability
        link2 = link_rates(dev)
        best = {k: max(link[k], link2[k]) for k in ("h2d_gbs", "d2h_gbs", "both_gbs")}
        bi, bo = host.h2d_bytes, host.d2h_bytes
        # the copies alone at the link rates: each direction at its own rate,
        # both together at the concurrent rate
        bound_ms = 1e3 * max(bi / (best["h2d_gbs"] * 1e9), bo / (best["d2h_gbs"] * 1e9),
                             (bi + bo) / (best["both_gbs"] * 1e9))
        e2e = {"value": round(job_throughput(n_job, ms_e2e), 3), "unit": UNIT,
               "ms_per_step": round(ms_e2e, 3), "ms_min": round(per[0], 3),
               "ms_median": round(per[len(per) // 2], 3), "steps": n_e2e,
               "h2d_bytes_per_step": bi, "d2h_bytes_per_step": bo, "group_mb": args.e2e_group_mb,
               "path": "iso_update_host: tensor groups copied in, updated and copied out on three streams",
               "link": {"before": link, "after": link2, "best": best},
               "link_bound_ms": round(bound_ms, 3), "of_link_bound": round(ms_e2e / bound_ms, 3)}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(name, budget_s=args.cpu_budget, rho=density)

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 3), "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 4),
            "higher_is_better": True, "scaling": "strong" if args.shard else "weak", "vs_baseline": None,
            "dtype": "bf16" if ckpt else "f32", "data": "synthetic (seeded, Qwen-shaped; no checkpoints)",
            "config": {"workload": name if not small else f"{name} (layers={args.layers}, widths/{args.scale})",
                       "description": desc, "params": n_params, "tensors": len(shapes),
                       "experts": K, "op": op, "density": density, "scope": scope,
                       "path": "fused single pass" if fused_pass(K, inputs, op, scope, args.two_pass)
                       else "separate passes",
                       "l2": "inputs larger than L2 (129 MB); no flush needed",
                       "parallelism": (f"tensor shards x{world}" if args.shard else f"replica x{world}")},
            "hbm_gbs_step": round(step_gbs, 1),
            "hbm_pct_of_8tbs_step": round(100 * step_gbs / NOMINAL_HBM_GBS, 1),
            "roofline": {"bound": "hbm", "kernel": dom, "achieved": round(achieved, 1), "peak": peak,
                         "peak_source": peak_src, "unit": "GB/s",
                         "frac": round(achieved / peak, 4) if peak else None, "traffic": traffic,
                         "traffic_source": "profiles/ ncu summary (DRAM bytes per param x params)"
                         if traffic is not None else "no ncu summary for the current kernel sources",
                         "algorithmic_bytes_per_launch": int(per_launch_bytes),
                         "avg_launch_ms": round(avg_ms, 4)},
            "kernels": {k: {"launches": v["launches"], "ms_per_step": round(v["ms_per_step"], 4)}
                        for k, v in sorted(kernels.items(), key=lambda kv: -kv[1]["ms_per_step"])},
            "gpu_launches": int(launches),
            "clocks": ck,
            "e2e": e2e,
            "cpu_baseline": cpu,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def pinned_flat(tensors, copy=True):
    """Page-locked host copies of a tensor list, as views of one buffer laid
    out back to back (each tensor starts on a 16-byte boundary)."""
    import torch
    dt = tensors[0].dtype
    step = 16 // tensors[0].element_size()
    offs, o = [], 0
    for t in tensors:
        offs.append(o)
        o += -(-t.numel() // step) * step
    buf = torch.empty(max(1, o), dtype=dt, pin_memory=True)
    views = [buf[a:a + t.numel()].view(t.shape) for a, t in zip(offs, tensors)]
    if copy:
        for v, t in zip(views, tensors):
            v.copy_(t)
    return views


def link_rates(dev, nbytes=2 << 30, reps=3):
    """Measured host<->device copy rates (GB/s) between page-locked host
    memory and HBM: one direction at a time, then both at once on two
    streams."""
    import torch
    h = [torch.empty(nbytes, dtype=torch.uint8, pin_memory=True) for _ in range(2)]
    d = [torch.empty(nbytes, dtype=torch.uint8, device=dev) for _ in range(2)]
    s1, s2 = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    cur = torch.cuda.current_stream(dev)

    def timed(fn):
        fn()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(cur)
        for _ in range(reps):
            fn()
        b.record(cur)
        torch.cuda.synchronize()
        return a.elapsed_time(b) / reps * 1e-3

    def both():
        s1.wait_stream(cur)
        s2.wait_stream(cur)
        with torch.cuda.stream(s1):
            d[0].copy_(h[0], non_blocking=True)
        with torch.cuda.stream(s2):
            h[1].copy_(d[1], non_blocking=True)
        cur.wait_stream(s1)
        cur.wait_stream(s2)

    t_in = timed(lambda: d[0].copy_(h[0], non_blocking=True))
    t_out = timed(lambda: h[1].copy_(d[1], non_blocking=True))
    t_both = timed(both)
    del h, d
    return {"h2d_gbs": round(nbytes / t_in / 1e9, 1), "d2h_gbs": round(nbytes / t_out / 1e9, 1),
            "both_gbs": round(2 * nbytes / t_both / 1e9, 1), "copy_bytes": nbytes}


def cpu_sample(name, seed=0):
    """A bounded, deterministic list of tensors of the workload (layer 0 first)."""
    import synth
    shapes_name = WORKLOADS[name][0]
    shapes = synth.qwen_shapes(shapes_name)
    order = list(range(1, 10)) + list(range(10, len(shapes)))   # layer 0, then onwards
    return shapes, order


def cpu_baseline(name, budget_s=15.0, seed=0, rho=None):
    """The oracle, as it stands, on a bounded sample of the workload: tensors
    are added in a fixed order until budget_s of single-thread CPU time."""
    import numpy as np
    import oracle
    import synth
    shapes_name, K, op, inputs, density, scope, _ = WORKLOADS[name]
    if rho is not None:
        density = rho
    if shapes_name == "sweep":
        return cpu_baseline_sweep(name, density, scope, seed)
    shapes, order = cpu_sample(name, seed)
    orc_op = {"ta": oracle.TA, "ties": oracle.TIES, "iso": oracle.ISO, "ram": oracle.RAM}[op]
    orc_scope = {"tensor": oracle.SCOPE_TENSOR, "block": oracle.SCOPE_BLOCK,
                 "global": oracle.SCOPE_GLOBAL}[scope]
    done, params, spent = [], 0, 0.0
    for q in order:
        s = shapes[q]
        if inputs == "ckpt_bf16":
            th0, th1 = synth.rl_update_set([s], seed=seed + q)
            a = [th0[0].view(-1).view(__import__("torch").int16).numpy().view(np.uint16).reshape(s[0], s[1])]
            ex = [[th1[0].view(-1).view(__import__("torch").int16).numpy().view(np.uint16).reshape(s[0], s[1])]]
        else:
            th0 = synth.base_weights([s], seed=seed + q)
            taus, _ = synth.merge_experts([s], seed=seed + q, K=K)
            a = [th0[0].view(-1).view(__import__("torch").int16).numpy().view(np.uint16).reshape(s[0], s[1])]
            ex = [[e[0].reshape(s[0], s[1]).numpy()] for e in taus]
        t = time.perf_counter()
        # the workload's scope on the sampled tensor (GLOBAL: the sample's own unit)
        oracle.merge(a, ex, orc_op, experts_are_deltas=(inputs != "ckpt_bf16"), density=density,
                     scope=orc_scope, is_1d=[s[2]])
        spent += time.perf_counter() - t
        params += s[0] * s[1]
        done.append(q)
        if spent >= budget_s:
            break
    return {"value": round(params / spent / 1e9, 6), "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"{len(done)} tensors of the workload ({params} params: tensor ids {done[0]}..{done[-1]} "
                      f"in layer order), timed on this host, single thread",
            "seconds": round(spent, 2)}


def cpu_baseline_sweep(name, rho, scope, seed=0):
    """The oracle on the whole density-sweep tensor (58.7 M entries)."""
    import numpy as np
    import torch
    import oracle
    import synth
    s = (4096, 14336, False)
    d = synth.density_sweep_delta(seed=seed, rho=rho)
    b = synth.base_weights([s], seed=seed)[0]
    a = b.view(torch.int16).numpy().view(np.uint16).reshape(s[0], s[1])
    x = d.view(torch.int16).numpy().view(np.uint16).reshape(s[0], s[1])
    sc = oracle.SCOPE_BLOCK if scope == "block" else oracle.SCOPE_TENSOR
    t = time.perf_counter()
    oracle.merge([a], [[x]], oracle.TIES, experts_are_deltas=True, density=rho, scope=sc)
    spent = time.perf_counter() - t
    return {"value": round(s[0] * s[1] / spent / 1e9, 6), "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"the whole 4096x14336 tensor ({scope} scope, rho={rho}), timed on this host, "
                      f"single thread", "seconds": round(spent, 2)}


def run_reference(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    name = args.workload
    rho = args.density if args.density is not None else WORKLOADS[name][4]
    per_step = max(2.0, args.cpu_budget / max(1, args.steps))
    for _ in range(args.warmup and 1):
        cpu_baseline(name, budget_s=0.5, rho=rho)
    vals = []
    for _ in range(args.steps):
        vals.append(cpu_baseline(name, budget_s=per_step, rho=rho))
    v = sum(x["value"] for x in vals) / len(vals)
    line = {
        "impl": "reference", "metric": METRIC, "value": round(v, 6), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64 values / f32 decisions", "data": "synthetic (seeded, Qwen-shaped)",
        "config": {"workload": name, "description": WORKLOADS[name][6]},
        "cpu_baseline": {"value": round(v, 6), "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": vals[-1]["sample"]},
        "e2e": {"value": round(v, 6), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["mine", "reference"], default="mine")
    ap.add_argument("--workload", choices=sorted(WORKLOADS) + ["frame_qwen7b_gate", "opt_qwen7b_gate"],
                    default="qwen7b_update")
    ap.add_argument("--frame-m", type=int, default=3584, help="frame workload: rows of the projection")
    ap.add_argument("--frame-n", type=int, default=18944, help="frame workload: columns of the projection")
    ap.add_argument("--experts", type=int, default=3, help="frame workload: RL experts merged")
    ap.add_argument("--two-pass", action="store_true",
                    help="run the K = 1 update as its two-pass form (count, then apply) "
                         "instead of the fused single pass")
    ap.add_argument("--shard", action="store_true",
                    help="N > 1: split one parameter set's tensors over the ranks (strong scaling) "
                         "instead of a replica per rank (weak scaling)")
    ap.add_argument("--density", type=float, default=None,
                    help="TopKMask density (default: the workload's own)")
    ap.add_argument("--compact-candidates", action="store_true",
                    help="K >= 2 TIES / ISO: the Gram and merge passes read the counting pass's "
                         "compact candidate values (iso_compact_candidates)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--e2e-group-mb", type=int, default=2048,
                    help="end-to-end leg: bytes (MiB) of one tensor group of the host-staged pipeline")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-budget", type=float, default=12.0)
    ap.add_argument("--clock-log", default=None,
                    help="keep the nvidia-smi clock samples of the timed region in this CSV "
                         "(default: a temporary file)")
    ap.add_argument("--layers", type=int, default=None,
                    help="decoder layers of the shape set (default: the model's own); "
                         "smaller cases are for profiling only")
    ap.add_argument("--scale", type=int, default=1,
                    help="divide every width of the shape set (profiling of small cases only)")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "mine":
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    elif args.workload == "frame_qwen7b_gate":
        run_frame(args)
    elif args.workload == "opt_qwen7b_gate":
        run_opt(args)
    else:
        run_mine(args)


if __name__ == "__main__":
    main()
