"""Benchmark: ms per full-model projected-Adam step on one GB300.

Workload: the 224 target matrices of a 32-layer Llama-2-7B-shaped model
(hidden 4096, MLP 11008) with the module-aware rank table q/k 512,
v/o/gate/up 1024, down 2048 (r_base 1024), block size 128, bf16 gradients,
fp32 weights and optimizer states; synthetic inputs (low-rank-plus-noise
gradients, random-normal weights).  One step is one moara_step_grouped call
over all 224 modules; the every-200-steps projector refresh is timed once and
added amortised (refresh_ms / 200).

value: device-timed ms per step (CUDA events on the launching stream, inputs
resident in HBM); e2e: the same step through the C ABI with the gradients
copied from pinned host memory each step and the device status word read
back.  roofline: the kernel with the largest share of step time, its
algorithmic bytes or flops per launch over its event-timed average launch.

`--impl reference` times the float64 oracle on the host cores instead.
"""

from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = "llama2_7b_full_module_aware"
METRIC = "ms per full-model projected-Adam step"
LR = 1e-3

# DRAM traffic (dram__bytes_read.sum + dram__bytes_write.sum) of one launch of
# each step kernel, from an ncu capture on the one-layer workload named here.
# A full-model launch processes the
# same kinds of tiles, so its traffic is scaled by the ratio of the kernel's
# algorithmic bytes (full model / captured workload).  Valid only for the
# kernel code with this fingerprint (SHA-1 of the step kernels' part of the
# source -- everything before the refresh GEMMs -- with `//` comments and
# blank lines removed); after any change there the roofline reports
# traffic = null until the counters are taken again.
TRAFFIC = {"source": "paper_2609_15037_gb300/csrc/tc.cu", "until": "// KR: bf16 tensor-core GEMM of the projector refresh",
           "sha1": "9a78720b38df49775e7f76e6b3052ea16cc22b4e",
           "workload": "llama7b_layer",
           "bytes": {"tc_decompose": 757951488, "tc_project": 1060206848, "tc_backproject": 1708868096}}


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            pk = json.load(f)
        return pk["hbm_gbs"], pk["bf16_tflops"], pk["bf16_tflops_sustained"], "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


def _dist():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def job_time_ms(elapsed_ms, world, device=None):
    """Time of the whole job's timed region: the maximum over ranks (each rank
    steps its own shard of the model's modules)."""
    if world <= 1:
        return float(elapsed_ms)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(elapsed_ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(step_ms, refresh_ms):
    """ms per full-model step of the whole job: the slowest rank's time for
    its shard of one step plus its refresh amortised over T = 200 steps (the
    ranks together step every module once)."""
    return step_ms + refresh_ms / 200.0


def shard_modules(n_modules, rank, world):
    """Indices of the modules rank `rank` owns: every world-th module, so that
    with 7 module types per layer each rank gets a mix of all types (the
    optimizer step needs no exchange between owners)."""
    return list(range(rank, n_modules, world))


class Clocks:
    """nvidia-smi sampling during the timed region."""

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        import tempfile
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={q}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            p = [x.strip() for x in line.split(",")]
            if len(p) < 9:
                continue
            try:
                sm.append(float(p[1]))
                mx.append(float(p[2]))
            except ValueError:
                continue
            for nm, v in zip(names, p[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        os.unlink(self.path)
        sm.sort()
        return {"sm_mhz": sm[len(sm) // 2] if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "samples": len(sm), "reasons": sorted(reasons)}


def _right(md, rule):
    """GaLore's smaller-side rule: a right projector for a tall weight."""
    return rule == "smaller" and md.m > md.n


def _algorithmic(mods, B, sb=4, rule="left"):
    """Algorithmic bytes and flops of one step over `mods` (Module list);
    sb: bytes per element of W and the direction moments (4 or 2); rule:
    projection side ("left", or "smaller": right projector when m > n)."""
    tot_b = tot_f = 0
    per = {"project": [0, 0], "backproject": [0, 0]}
    for md in mods:
        m, n, r = md.m, md.n, md.r
        k = -(-n // B)
        # R is r x n, or m x r with a right projector (n x r)
        rc, pr = (m, n) if _right(md, rule) else (n, m)
        # minimum traffic of one fused pass: G read (bf16), W read+write,
        # direction moments read+write, P read once (bf16), magnitude moments
        tot_b += 2 * m * n + 2 * sb * m * n + 4 * sb * r * rc + 2 * pr * r + 16 * m * k
        tot_f += 4 * m * r * n
        per["project"][1] += 2 * m * r * n
        per["backproject"][1] += 2 * m * r * n
    return tot_b, tot_f, per


def _kernel_bytes(mods, B, tc, sb=4, rule="left"):
    """Algorithmic bytes per step of each step kernel as built.

    tensor-core path: tc_decompose reads G (bf16), writes V (bf16) and updates
    the magnitude moments (read+write) and dM; tc_project reads V, P (bf16) and
    the direction moments (read+write) and writes N (bf16); tc_backproject
    reads and writes W and reads N, P (bf16) and dM.  fp32 path: decompose
    reads G and writes the block scales, project reads G, the scales, P (fp32)
    and the moments and writes N (fp32), backproject as above with fp32 N, P.
    """
    kb = {}
    for md in mods:
        m, n, r = md.m, md.n, md.r
        k = -(-n // B)
        if tc:
            rc, pr = (m, n) if _right(md, rule) else (n, m)   # R: r x rc; projector: pr x r
            add = {"tc_decompose": 2 * m * n + 2 * m * n + 20 * m * k,
                   "tc_project": 2 * m * n + 2 * pr * r + 4 * sb * r * rc + 2 * r * rc,
                   "tc_backproject": 2 * sb * m * n + 2 * r * rc + 2 * pr * r + 4 * m * k}
        else:
            add = {"decompose": 2 * m * n + 20 * m * k + 4 * m * k,
                   "project": 2 * m * n + 4 * m * k + 4 * m * r + 16 * r * n + 4 * r * n,
                   "backproject": 8 * m * n + 4 * r * n + 4 * m * r + 4 * m * k}
        for key, v in add.items():
            kb[key] = kb.get(key, 0) + v
    return kb


def _code_sha1(path, until=None):
    """SHA-1 of a C++/CUDA source (up to the first line that starts with
    `until`, if given) with `//` comments and blank lines removed."""
    import hashlib
    lines = []
    with open(path, encoding="utf-8") as f:
        for raw in f:
            if until is not None and raw.startswith(until):
                break
            ln = raw.split("//", 1)[0].strip()
            if ln:
                lines.append(ln)
    return hashlib.sha1("\n".join(lines).encode()).hexdigest()


def _traffic(kernel, workload):
    """Per-launch DRAM bytes of `kernel` at `workload` (from the captured
    counters, scaled by algorithmic bytes), or None."""
    import hashlib
    import synth
    if TRAFFIC["sha1"] is None or kernel not in TRAFFIC["bytes"]:
        return None
    if _code_sha1(os.path.join(ROOT, TRAFFIC["source"]), TRAFFIC["until"]) != TRAFFIC["sha1"]:
        return None
    cap = synth.workload(TRAFFIC["workload"])
    cur = synth.workload(workload)
    scale = (_kernel_bytes(cur["modules"], cur["block_size"], True)[kernel] /
             _kernel_bytes(cap["modules"], cap["block_size"], True)[kernel])
    return int(TRAFFIC["bytes"][kernel] * scale)


def _rank_summary(mods):
    """Ranks by module type, e.g. 'q 512, k 512, v 1024, ...' (first layer)."""
    seen = {}
    for md in mods:
        seen.setdefault(md.mtype, md.r)
    return ", ".join(f"{t} {r}" for t, r in seen.items())


def run_gpu(args):
    import torch
    import paper_2609_15037_gb300 as M
    import synth

    rank, world, local = _dist()
    torch.cuda.set_device(local)
    dev = torch.device(f"cuda:{local}")
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    wl = synth.workload(args.workload)
    all_mods = wl["modules"]
    # N > 1: each rank owns every world-th module and steps only those
    sel = shard_modules(len(all_mods), rank, world)
    mods = [all_mods[i] for i in sel]
    B = wl["block_size"]
    hp = M.moara_default_hparams()
    hp.block_size = B
    hp.adam_eps = wl["adam_eps"]
    hp.clip_norm = args.clip_norm
    hp.state_dtype = M.MOARA_DTYPE_BF16 if args.state_dtype == "bf16" else M.MOARA_DTYPE_F32
    sbytes = 2 if args.state_dtype == "bf16" else 4
    hp.proj_rule = M.MOARA_PROJ_SMALLER if args.proj_rule == "smaller" else M.MOARA_PROJ_LEFT
    g = M.MoaraGroup(hp, device=local, refresh_workspace_bytes=int(args.refresh_ws_gb * (1 << 30)))
    stream = torch.cuda.current_stream(dev)
    grads = []
    for i, md in enumerate(mods):
        g.add(md.m, md.n, md.r, "bf16")
        with torch.no_grad():
            g.modules[i].W.normal_(0.0, 0.02)
        grads.append(synth.lowrank_grad_torch(md.m, md.n, wl["signal_rank"], wl["sigma0"],
                                              wl["noise"], 1, seed=0, module=sel[i],
                                              noise_rel=wl["noise_rel"], device=dev))
    torch.cuda.synchronize()
    ids = list(g.ids)
    gptr = [x.data_ptr() for x in grads]
    cs = stream.cuda_stream

    # projector refresh (once, timed; amortised over T = 200 steps)
    g.ensure_refresh_workspace()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    M.moara_refresh_projector(g.ctx, ids, gptr, cs)
    t1.record(stream)
    torch.cuda.synchronize()
    refresh_ms = t0.elapsed_time(t1)

    # warm-up
    step = 1
    for _ in range(args.warmup):
        M.moara_step_grouped(g.ctx, ids, gptr, step, LR, False, cs)
        step += 1
    torch.cuda.synchronize()

    # timed region (device time, CUDA events on the launching stream)
    M.moara_profile_read(g.ctx)
    M.moara_profile_enable(g.ctx, True)
    launches0 = M.moara_launch_count(g.ctx)
    clocks = Clocks(local)
    clocks.start()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        M.moara_step_grouped(g.ctx, ids, gptr, step, LR, False, cs)
        step += 1
    ev1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    clk = clocks.stop()
    launches = M.moara_launch_count(g.ctx) - launches0
    M.moara_profile_enable(g.ctx, False)
    prof = M.moara_profile_read(g.ctx)
    elapsed = job_time_ms(ev0.elapsed_time(ev1), world, dev)
    step_ms = elapsed / args.steps
    status = M.moara_get_device_status(g.ctx, cs)

    # alignment diagnostic S(W, t) over every module (a profiling-step call,
    # outside the step; it reuses the modules' workspaces, which the next
    # step rewrites): one untimed call, then the mean of three
    a_sel = list(range(len(mods)))
    a_ids, a_ptr = [ids[k] for k in a_sel], [gptr[k] for k in a_sel]
    S_dev = torch.empty(max(1, len(a_ids)), dtype=torch.float32, device=dev)
    M.moara_alignment(g.ctx, a_ids, a_ptr, S_dev.data_ptr(), cs)
    a0 = torch.cuda.Event(enable_timing=True)
    a1 = torch.cuda.Event(enable_timing=True)
    a0.record(stream)
    for _ in range(3):
        M.moara_alignment(g.ctx, a_ids, a_ptr, S_dev.data_ptr(), cs)
    a1.record(stream)
    torch.cuda.synchronize()
    align_ms = a0.elapsed_time(a1) / 3
    S_host = S_dev.cpu().numpy()
    status |= M.moara_get_device_status(g.ctx, cs)

    # end to end through the C ABI with host buffers: every step uploads its
    # gradients from page-locked host memory (moara_step_grouped_host overlaps
    # the chunked upload with the step kernels) and reads the device status
    # word back
    host = [torch.empty(x.shape, dtype=x.dtype, pin_memory=True) for x in grads]
    for h, x in zip(host, grads):
        h.copy_(x)
    hptr = [h.data_ptr() for h in host]
    e2e_steps = max(1, min(args.steps, 10))
    chunk = int(args.chunk_mb) << 20
    # clipping needs every gradient on the device before the first update, so
    # the clipped step uploads all of them (plain copies) and then steps
    via_host_call = args.clip_norm <= 0

    def e2e_step(st):
        if via_host_call:
            M.moara_step_grouped_host(g.ctx, ids, hptr, st, LR, False, chunk, cs)
        else:
            for h, x in zip(host, grads):
                x.copy_(h, non_blocking=True)
            M.moara_step_grouped(g.ctx, ids, gptr, st, LR, False, cs)

    for _ in range(max(1, args.warmup)):   # staging allocation, then the same warm-up as the device timing
        e2e_step(step)
        step += 1
    torch.cuda.synchronize()
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(e2e_steps + 1)]
    evs[0].record(stream)
    e2e_status = 0
    for k in range(e2e_steps):
        e2e_step(step)
        step += 1
        e2e_status |= M.moara_get_device_status(g.ctx, cs)
        evs[k + 1].record(stream)
    torch.cuda.synchronize()
    e2e_ms = job_time_ms(evs[0].elapsed_time(evs[-1]), world, dev) / e2e_steps
    e2e_each = sorted(evs[k].elapsed_time(evs[k + 1]) for k in range(e2e_steps))
    e2e_median = job_time_ms(e2e_each[len(e2e_each) // 2], world, dev)
    h2d = sum(x.numel() * x.element_size() for x in grads)
    # the host link alone: the same bytes copied into the device gradients
    torch.cuda.synchronize()
    # (best of three: the first pass over the pinned buffers runs slower)
    c0 = torch.cuda.Event(enable_timing=True)
    c1 = torch.cuda.Event(enable_timing=True)
    h2d_gbs = 0.0
    for _ in range(3):
        c0.record(stream)
        for h, x in zip(host, grads):
            x.copy_(h, non_blocking=True)
        c1.record(stream)
        torch.cuda.synchronize()
        h2d_gbs = max(h2d_gbs, h2d / (c0.elapsed_time(c1) * 1e-3) / 1e9)

    hbm, bf16_peak, bf16_sus, peak_src = _peaks()
    alg_bytes, alg_flops, _ = _algorithmic(mods, B, sbytes, args.proj_rule)
    total_ms = step_ms + refresh_ms / 200.0
    roof_ms = max(alg_bytes / (hbm * 1e9), alg_flops / (bf16_sus * 1e12)) * 1e3
    # the refresh's product flops: 2q + 2 products of V (m x n) with an
    # n x l or m x l basis, l = min(r + p, m, n), at 2 m n l flops each
    rf_flops = 0.0
    for md in mods:
        lw = min(md.r + hp.oversample, md.m, md.n)
        rf_flops += (2 * hp.power_iters + 2) * 2.0 * md.m * md.n * lw
    rf_roof_ms = rf_flops / (bf16_sus * 1e12) * 1e3

    # dominant kernel
    used_tc = prof["tc_project"][1] > 0
    kbytes = _kernel_bytes(mods, B, used_tc, sbytes, args.proj_rule)
    names = ["decompose", "project", "backproject", "tc_decompose", "tc_project", "tc_backproject"]
    dom = max(names, key=lambda k: prof[k][0])
    dom_ms = prof[dom][0] / max(prof[dom][1], 1)
    n_launch_per_step = max(prof[dom][1] // args.steps, 1)
    flops_dom = alg_flops / 2 / n_launch_per_step
    if dom in ("project", "backproject"):
        # fp32 SIMT GEMM: bound by the FP32 FMA pipes
        alu_peak = 152 * 128 * 2 * 2.07e9 / 1e12
        achieved = flops_dom / (dom_ms * 1e-3) / 1e12
        roof = {"bound": "alu", "achieved": round(achieved, 2), "peak": round(alu_peak, 1),
                "unit": "TFLOP/s", "frac": round(achieved / alu_peak, 4), "traffic": None,
                "kernel": dom, "peak_source": "152 SMs x 128 FP32 lanes x 2 x 2.07 GHz"}
    elif dom in ("tc_project", "tc_backproject") and \
            flops_dom / (bf16_sus * 1e12) >= kbytes[dom] / n_launch_per_step / (hbm * 1e9):
        # the kernel's own roof is the tensor pipe: its flops at the sustained
        # bf16 rate take longer than its bytes at the copy bandwidth
        achieved = flops_dom / (dom_ms * 1e-3) / 1e12
        # the counters were taken with fp32 states and left projectors
        tr = _traffic(dom, args.workload) if (sbytes == 4 and args.proj_rule == "left") else None
        roof = {"bound": "tensor", "achieved": round(achieved, 1), "peak": bf16_sus,
                "unit": "TFLOP/s", "frac": round(achieved / bf16_sus, 4),
                "traffic": None if tr is None else int(tr / n_launch_per_step),
                "kernel": dom, "peak_source": f"bf16_tflops_sustained ({peak_src})",
                "hbm_frac": round(kbytes[dom] / n_launch_per_step / (dom_ms * 1e-3) / 1e9 / hbm, 4)}
    else:
        by = kbytes[dom] / n_launch_per_step
        achieved = by / (dom_ms * 1e-3) / 1e9
        # the counters were taken with fp32 states and left projectors
        tr = _traffic(dom, args.workload) if (sbytes == 4 and args.proj_rule == "left") else None
        roof = {"bound": "hbm", "achieved": round(achieved, 1), "peak": hbm, "unit": "GB/s",
                "frac": round(achieved / hbm, 4), "traffic": None if tr is None else int(tr / n_launch_per_step),
                "kernel": dom, "peak_source": f"hbm_gbs ({peak_src})"}

    kernels = {}
    overlap = prof["tc_decompose_overlap"][1] > 0
    for k in names:
        if prof[k][1] == 0:
            continue
        ms = prof[k][0] / args.steps
        kernels[k] = {"ms_per_step": round(ms, 4), "launches_per_step": prof[k][1] / args.steps,
                      "share": round(prof[k][0] / max(sum(prof[x][0] for x in names), 1e-9), 4),
                      "alg_gbs": round(kbytes.get(k, 0) / (ms * 1e-3) / 1e9, 1)}
        if k in ("tc_project", "tc_backproject"):
            # each product kernel's algorithmic flops (half the step's) and its
            # own bytes against the sustained bf16 rate and the copy bandwidth
            kernels[k]["tensor_frac"] = round(alg_flops / 2 / (ms * 1e-3) / 1e12 / bf16_sus, 4)
            kernels[k]["hbm_frac"] = round(kbytes.get(k, 0) / (ms * 1e-3) / 1e9 / hbm, 4)
    if overlap:
        # the decomposition of all but the first module part runs on the
        # library's auxiliary stream, concurrent with K1 / K2: its event time
        # overlaps theirs and its bytes are split between the two entries
        kernels["tc_decompose"]["alg_gbs"] = None
        kernels["tc_decompose_overlap"] = {
            "ms_per_step": round(prof["tc_decompose_overlap"][0] / args.steps, 4),
            "launches_per_step": prof["tc_decompose_overlap"][1] / args.steps,
            "share": None, "alg_gbs": None, "stream": "auxiliary (concurrent with tc_project / tc_backproject)"}
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(args, budget_s=args.cpu_seconds)
    out = {
        "metric": METRIC, "value": round(job_value(step_ms, refresh_ms), 4), "unit": "ms",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(total_ms, 4), "higher_is_better": False,
        "scaling": "strong" if world > 1 else "weak",
        "vs_baseline": None,
        "dtype": "bf16" if used_tc else "f32",
        "data": "synthetic",
        "config": {"workload": args.workload, "modules": len(all_mods), "block_size": B,
                   "ranks": _rank_summary(mods),
                   "precision": (("bf16 MMA operands (G, V, P, N), fp32 accumulation and elementwise; "
                                  + ("bf16 W and direction states, fp32 magnitude states" if sbytes == 2
                                     else "fp32 W and states")) if used_tc
                                 else "fp32 SIMT (bf16 G read as is)"),
                   "l2": "inputs larger than L2 (no flush needed)",
                   "parallelism": f"module-sharded x{world} (no exchange)" if world > 1 else "single GPU",
                   "clip_norm": args.clip_norm, "state_dtype": args.state_dtype,
                   "proj_rule": args.proj_rule},
        "step_ms_no_refresh": round(step_ms, 4),
        "clip_norm_ms": round(prof["clip_norm"][0] / args.steps, 4) if prof["clip_norm"][1] else None,
        "refresh_ms": round(refresh_ms, 2), "refresh_amortised_ms": round(refresh_ms / 200.0, 4),
        "refresh_roofline": {"flops": rf_flops, "roofline_ms": round(rf_roof_ms, 2),
                             "frac": round(rf_roof_ms / refresh_ms, 4) if refresh_ms > 0 else None,
                             "basis": f"(2q+2)*2*m*n*(r+p) with q = {hp.power_iters}, p = {hp.oversample}, "
                                      f"at the sustained bf16 rate"},
        "hbm_gbs_algorithmic": round(alg_bytes / (step_ms * 1e-3) / 1e9, 1),
        "step_roofline": {"alg_bytes": alg_bytes, "alg_flops": alg_flops,
                          "roofline_ms": round(roof_ms, 3),
                          "frac": round(roof_ms / step_ms, 4),
                          "peaks": f"hbm {hbm} GB/s, bf16 {bf16_sus} TFLOP/s sustained ({peak_src})"},
        "roofline": roof,
        "kernels": kernels,
        "e2e": {"value": round(job_value(e2e_median, refresh_ms), 4), "unit": "ms",
                "step_ms_mean": round(e2e_ms, 3),
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": 4,
                "h2d_gbs_link": round(h2d_gbs, 1),
                "link_floor_ms": round(h2d / (h2d_gbs * 1e9) * 1e3, 3),
                "step_ms_median": round(e2e_median, 3), "steps": e2e_steps,
                "path": "moara_step_grouped_host" if via_host_call else "host-to-device copies + moara_step_grouped"},
        "alignment": {"ms": round(align_ms, 3), "modules": len(a_ids),
                      "flops": int(4 * sum(mods[k].m * mods[k].n * mods[k].r for k in a_sel)),
                      "tflops": round(4 * sum(mods[k].m * mods[k].n * mods[k].r for k in a_sel)
                                      / max(align_ms * 1e-3, 1e-9) / 1e12, 1),
                      "S_mean": round(float(S_host[:len(a_ids)].mean()), 4) if a_ids else None},
        "gpu_launches": int(launches),
        "device_status": status | e2e_status,
        "clocks": clk,
    }
    if cpu is not None:
        out["cpu_baseline"] = cpu
    if rank == 0:
        print(json.dumps(out), flush=True)
    g.close()
    if world > 1:
        torch.distributed.destroy_process_group()


def _oracle_layer_sample(wl, layer_modules, seed=0, rule="left", state_bf16=False):
    """Oracle step on the seven modules of one decoder layer (float64)."""
    import numpy as np
    from oracle import moara_ref as o
    hp = o.Hparams(block_size=wl["block_size"], adam_eps=wl["adam_eps"], proj_rule=rule, state_bf16=state_bf16)
    rng = np.random.default_rng(seed)
    states, grads = [], []
    for md in layer_modules:
        W = rng.standard_normal((md.m, md.n)) * 0.02
        right = _right(md, rule)
        P = np.linalg.qr(rng.standard_normal((md.n if right else md.m, md.r)))[0]
        states.append(o.init_state(W, md.r, wl["block_size"], P=P, proj_rule=rule))
        grads.append(rng.standard_normal((md.m, md.n)) * 1e-3)
    return states, grads, hp


def _oracle_module_ms(args, threads):
    """Oracle step time (best of two) of layer 0's first module, in a child
    process whose BLAS runs `threads` threads (the thread count is fixed when
    NumPy loads its BLAS, hence the child)."""
    rule = getattr(args, "proj_rule", "left")
    sb = getattr(args, "state_dtype", "f32") == "bf16"
    code = "\n".join([
        "import sys, time, json",
        f"sys.path.insert(0, {ROOT!r})",
        "import bench, synth",
        "from oracle import moara_ref as o",
        f"wl = synth.workload({args.workload!r})",
        "md = [m for m in wl['modules'] if m.name.startswith('layer0.')][0]",
        f"st, gr, hp = bench._oracle_layer_sample(wl, [md], rule={rule!r}, state_bf16={sb!r})",
        "best = 1e30",
        "for t in (1, 2):",
        "    t0 = time.perf_counter()",
        "    st[0] = o.step(st[0], gr[0], t, bench.LR, hp, refresh=False)",
        "    best = min(best, time.perf_counter() - t0)",
        "print(json.dumps({'ms': best * 1e3, 'shape': f'{md.m}x{md.n} r {md.r}'}))",
    ])
    env = dict(os.environ, OMP_NUM_THREADS=str(threads), OPENBLAS_NUM_THREADS=str(threads),
               MKL_NUM_THREADS=str(threads))
    try:
        res = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True,
                             timeout=300, cwd=ROOT)
        return json.loads(res.stdout.strip().splitlines()[-1])
    except Exception:
        return None


def cpu_baseline(args, budget_s=20.0):
    """The oracle as it stands, one 7B decoder layer per sample, scaled to the
    full model (x layers).  Runs in this process on the host cores."""
    import numpy as np
    from oracle import moara_ref as o
    import synth
    wl = synth.workload(args.workload)
    layer = [md for md in wl["modules"] if md.name.startswith("layer0.")]
    layers = len(wl["modules"]) // len(layer)
    states, grads, hp = _oracle_layer_sample(wl, layer, rule=getattr(args, "proj_rule", "left"),
                                             state_bf16=getattr(args, "state_dtype", "f32") == "bf16")
    times = []
    t_start = time.time()
    t = 1
    while True:
        t0 = time.perf_counter()
        for i in range(len(layer)):
            states[i] = o.step(states[i], grads[i], t, LR, hp, refresh=False)
        times.append(time.perf_counter() - t0)
        t += 1
        if time.time() - t_start > budget_s or len(times) >= 3:
            break
    per_layer = min(times)
    try:
        cores = len(os.sched_getaffinity(0))
    except Exception:
        cores = os.cpu_count()
    threads = os.environ.get("OMP_NUM_THREADS") or os.environ.get("OPENBLAS_NUM_THREADS") or str(cores)
    out = {"value": round(per_layer * layers * 1e3, 1), "unit": "ms", "cores": int(threads),
           "kind": "oracle",
           "sample": f"one decoder layer (7 modules) of the {len(wl['modules'])}-matrix model, "
                     f"float64 NumPy step without refresh, best of {len(times)}, x{layers} layers"}
    # the same oracle on one module at one BLAS thread and at all of them
    one = _oracle_module_ms(args, 1)
    allc = _oracle_module_ms(args, int(threads))
    if one is not None and allc is not None:
        out["one_module"] = {"shape": one["shape"], "ms_1_thread": round(one["ms"], 1),
                             "ms_all_threads": round(allc["ms"], 1), "threads": int(threads)}
    return out


def run_reference(args):
    """Times the oracle on the host cores (rank 0 only)."""
    rank, world, _ = _dist()
    if rank != 0:
        return
    import synth
    from oracle import moara_ref as o
    wl = synth.workload(args.workload)
    layer = [md for md in wl["modules"] if md.name.startswith("layer0.")]
    layers = len(wl["modules"]) // len(layer)
    states, grads, hp = _oracle_layer_sample(wl, layer, rule=getattr(args, "proj_rule", "left"),
                                             state_bf16=getattr(args, "state_dtype", "f32") == "bf16")
    t = 1
    for _ in range(args.warmup):
        for i in range(len(layer)):
            states[i] = o.step(states[i], grads[i], t, LR, hp, refresh=False)
        t += 1
    t0 = time.perf_counter()
    for _ in range(args.steps):
        for i in range(len(layer)):
            states[i] = o.step(states[i], grads[i], t, LR, hp, refresh=False)
        t += 1
    per_layer = (time.perf_counter() - t0) / args.steps
    val = per_layer * layers * 1e3
    try:
        cores = len(os.sched_getaffinity(0))
    except Exception:
        cores = os.cpu_count()
    out = {"impl": "reference", "metric": METRIC, "value": round(val, 1), "unit": "ms",
           "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
           "ms_per_step": round(val, 1), "higher_is_better": False, "scaling": "weak",
           "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": {"workload": args.workload, "modules": len(wl["modules"]),
                      "block_size": wl["block_size"]},
           "cpu_baseline": {"value": round(val, 1), "unit": "ms", "cores": cores,
                            "kind": "oracle",
                            "sample": f"each step: one decoder layer (7 modules) in float64 "
                                      f"NumPy, x{layers} layers, no refresh"},
           "e2e": {"value": round(val, 1), "unit": "ms", "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=25)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="gpu", choices=["gpu", "reference"])
    ap.add_argument("--workload", default=WORKLOAD)
    ap.add_argument("--cpu-seconds", type=float, default=20.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--refresh-ws-gb", type=float, default=44.0)
    ap.add_argument("--state-dtype", default="f32", choices=["f32", "bf16"],
                    help="W and direction moments in fp32 (the workload's definition) or bf16 (the paper's runs)")
    ap.add_argument("--proj-rule", default="left", choices=["left", "smaller"],
                    help="left projector for every weight (the workload's definition) or GaLore's smaller-side rule")
    ap.add_argument("--clip-norm", type=float, default=0.0,
                    help="global-norm gradient clipping threshold (0: off, as in the workload's definition)")
    ap.add_argument("--chunk-mb", type=int, default=256,
                    help="gradient chunk of the host-gradient step (e2e)")
    args = ap.parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
