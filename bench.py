#!/usr/bin/env python
"""Benchmark of the BOM (Backpropagated Output Momentum) hot path on GB300.

One timed step = one pass of the whole path over one batch: backbone forward
(two SwiGLU MLP sublayers), logits + cross-entropy statistics, residuals, s_t,
the q_t EMA, the head and backbone backward with the reprojection folded in,
and the BOM-AdamW update of every parameter (fused into the epilogues of the
weight-gradient GEMMs; --separate-update runs it as its own pass).  The workload is the largest
single-GPU configuration: 16384 tokens, d = 2048, ffn = 8192, vocabulary 32000,
166,199,296 parameters (fp32 master weights, bf16 compute copies).

Prints ONE JSON line (rank 0).  Besides the headline tokens/s it carries the
roofline of the dominant kernel, the end-to-end number through host buffers,
the clocks sampled during the timed region, and the oracle timed on the host
cores on a bounded sample (cpu_baseline).  The headline comes from untraced
steps; the per-kernel split (and the dominant kernel's launch time) from
separate steps with CUDA events around every launch.  Sub-measurements of the
same metric family ride along: the head-only LM output block (8192 x 768 x
50257) in tokens/s and as a fraction of the bf16 peak, the update alone over
10M, 125M and 1e9 elements in GB/s (both also as keys of the roofline
object), BOM-Adam-mini, the clipped update, the telemetry step, the RMSNorm
variant and the two small configurations.

--impl reference times the fp64 CPU oracle on the host cores instead (the
only reference implementation this method has here).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

from paper_2609_36738_gb300 import inputs as I  # noqa: E402

METRIC = "BOM step tokens/s (fused head+reprojection) and update GB/s vs GB300 roofline"
# lr 1e-4: the synthetic batch repeats every step and the SwiGLU stack has no
# normalisation, so a larger constant rate drives the logits to overflow
# within the few dozen steps a run takes.
LR, WD, LAM, B1, B2, EPS = 1e-4, 0.1, 0.5, 0.9, 0.999, 1e-8
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def _args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=50)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--workload", default="lm_mlp_bf16")
    p.add_argument("--no-extra", action="store_true", help="skip the head-only and update sub-measurements")
    p.add_argument("--parallel", default=None, choices=["replicas", "dp", "vocab"],
                   help="replicas: independent steps per rank (the default on one GPU); dp: the data-parallel "
                        "step, rows split across ranks, one all-reduce of the V + 3 exchange sums and one of "
                        "the gradient shares, then the update (the default under torchrun); vocab: the head's "
                        "columns split across ranks, every rank with the whole batch, an all-gather of the row "
                        "log-sum-exp parts and an all-reduce of the head's input cotangent, then the update")
    p.add_argument("--no-cpu", action="store_true", help="skip the cpu_baseline leg")
    p.add_argument("--separate-update", action="store_true",
                   help="run bom_update after bom_step instead of the update fused into the step")
    p.add_argument("--tokens", type=int, default=0,
                   help="smaller batch of the same workload (profiling captures); 0 = the workload's own")
    return p.parse_args()


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        d = json.load(open(path))
        return {k: float(d[k]) for k in FALLBACK_PEAKS}, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def _workload_desc(wl):
    if wl.name == "lm_mlp_bf16":
        return ("LM output block + 2 SwiGLU MLP sublayers: 16384 tokens, d=2048, ffn=8192, vocab 32000, "
                "full BOM backward and BOM-AdamW update over 166,199,296 params")
    if wl.name == "tiny_mlp_f32":
        return "tiny MLP classifier, fp32: 64 -> 128 (GELU) -> 10 classes, batch 32"
    if wl.name == "vision_head_bf16":
        return "vision-style classifier head, bf16: 768 -> 3072 -> 768 (GELU) -> 1000 classes, batch 256"
    return wl.name


# --------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi samples every 50 ms; only the samples taken between mark_start()
    and mark_end() (the timed steps) enter the summary."""
    FIELDS = ["timestamp", "clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.hw_slowdown",
              "clocks_event_reasons.hw_thermal_slowdown", "clocks_event_reasons.sw_thermal_slowdown",
              "clocks_event_reasons.sw_power_cap"]

    def __init__(self, gpu_id):
        self.gpu_id = gpu_id
        self.proc = None
        self.t0 = self.t1 = None
        self.path = os.path.join("/tmp", f"bom_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={','.join(self.FIELDS)}", "--format=csv,noheader,nounits",
                 "-i", str(self.gpu_id), "-lms", "50"], stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def mark_start(self):
        self.t0 = time.time()

    def mark_end(self):
        self.t1 = time.time()

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.fh.close()
        import datetime
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        rows = []
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                ts = datetime.datetime.strptime(parts[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                rows.append((ts, float(parts[1]), float(parts[2]), float(parts[3]), parts[4:8]))
            except ValueError:
                continue
        os.remove(self.path)
        inside = [r for r in rows if self.t0 is not None and self.t1 is not None and self.t0 <= r[0] <= self.t1]
        use = inside if inside else rows
        reasons = set()
        for r in use:
            for nm, v in zip(names, r[4]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        sm = [r[1] for r in use]
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(r[2] for r in use) if use else None,
                "sm_mhz_min": min(sm) if sm else None,
                "power_w_median": statistics.median([r[3] for r in use]) if use else None,
                "reasons": sorted(reasons), "samples": len(sm),
                "window": "timed steps only" if inside else "whole sampler run (no sample inside the timed steps)"}


# --------------------------------------------------------------------- CPU oracle legs
_ORACLE_INPUTS = {}


def oracle_sample(wl, seed=0, n_rows=None, budget_s=15.0):
    """Times the fp64 oracle on a bounded sample of the workload: one BOM step on
    the first n_rows rows of the batch through the full-size network, plus the
    update over the same fraction of the parameters.  Returns (tokens/s, desc)."""
    import oracle as O
    key = (wl.name, seed)
    if key not in _ORACLE_INPUTS:
        params = I.init_params(wl, seed)
        p64 = [I.bf16_to_f64(p) if wl.dtype == "bf16" else p.astype(np.float64) for p in params]
        x, y = I.make_batch(wl, seed, 1)
        xs = I.bf16_to_f64(x) if wl.dtype == "bf16" else x.astype(np.float64)
        _ORACLE_INPUTS.clear()
        _ORACLE_INPUTS[key] = (p64, xs, y)
    p64, xs, y = _ORACLE_INPUTS[key]
    layers = [(l.kind, l.d_in, l.d_out, l.has_bias) for l in wl.layers]
    n = n_rows or 16
    while True:
        t0 = time.perf_counter()
        out = O.bom_step(layers, wl.head_bias, p64, xs[:n], y[:n], np.zeros(wl.vocab), 1)
        frac = n / wl.n_rows
        for k, p in enumerate(p64):
            m = max(1, int(p.size * frac))
            O.bom_update(p.ravel()[:m], out["u"][k].ravel()[:m], np.zeros(m), LR, WD, 1, B2, EPS)
        dt = time.perf_counter() - t0
        if n_rows is not None or dt > budget_s / 4 or n * 2 > wl.n_rows:
            break
        n *= 2
    desc = (f"{n} of {wl.n_rows} rows through the full-size network (forward, task-space pass, the "
            f"oracle's three reverse passes for g, h and u) + the update over {n}/{wl.n_rows} of the "
            f"{wl.n_params()} parameters; fp64 numpy")
    return n / dt, desc, n


def run_reference(a):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    wl = I.WORKLOADS[a.workload]
    cores = os.cpu_count()
    # rows per step sized so that warm-up and timed steps together take about 1-2 minutes
    _, desc, n = oracle_sample(wl, budget_s=min(8.0, 200.0 / max(1, a.steps + a.warmup)))
    for _ in range(a.warmup):
        oracle_sample(wl, n_rows=n)
    vals = []
    t_all = time.perf_counter()
    for _ in range(a.steps):
        v, _, _ = oracle_sample(wl, n_rows=n)
        vals.append(v)
    total = time.perf_counter() - t_all
    value = a.steps * n / total
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": a.steps, "warmup": a.warmup, "ms_per_step": 1e3 * total / a.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": _workload_desc(wl), "sample_rows_per_step": n},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle", "sample": desc},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------------- GPU leg
def main():
    a = _args()
    if a.impl == "reference":
        return run_reference(a)
    import torch

    from paper_2609_36738_gb300 import bom as B
    from paper_2609_36738_gb300 import build as builder

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    if rank == 0:
        builder.build()
    if dist is not None:
        dist.barrier()
    B.lib()
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream()
    peaks, peak_src = _peaks()

    # ---------------------------------------------------------------- workload state
    wl = I.WORKLOADS[a.workload]
    if a.tokens:
        import dataclasses
        wl = dataclasses.replace(wl, n_rows=a.tokens)
    mode = a.parallel or ("dp" if world > 1 else "replicas")
    dp, vocab_par = mode == "dp", mode == "vocab"
    # data- and vocabulary-parallel ranks hold one model; replicas are independent models
    params_np = I.init_params(wl, seed=rank if mode == "replicas" else 0)
    V_total, v_first, wl_model = wl.vocab, 0, wl
    if vocab_par:   # this rank's rows of the head (and of its bias)
        import dataclasses
        cols = np.array_split(np.arange(V_total), world)[rank]
        v_first = int(cols[0])
        hw = len(params_np) - (2 if wl.head_bias else 1)
        params_np = list(params_np)
        for k in range(hw, len(params_np)):
            params_np[k] = np.ascontiguousarray(params_np[k][v_first:v_first + cols.size])
        wl_model = dataclasses.replace(wl, vocab=int(cols.size))
    shapes = [s for _, s, _ in wl_model.param_shapes()]
    sizes = [int(np.prod(s)) for s in shapes]
    offs = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int64)
    # pad every tensor to 8 elements so each view is 16-byte aligned
    offs_al = np.concatenate([[0], np.cumsum([(s + 7) // 8 * 8 for s in sizes])]).astype(np.int64)
    P = int(offs_al[-1])
    bf16 = wl.dtype == "bf16"
    master = torch.zeros(P, dtype=torch.float32, device=dev)
    shadow = torch.zeros(P, dtype=torch.bfloat16 if bf16 else torch.float32, device=dev)
    gradf = torch.zeros(P, dtype=shadow.dtype, device=dev)
    vstate = torch.zeros(P, dtype=torch.float32, device=dev)
    for k, p in enumerate(params_np):
        o = int(offs_al[k])
        vals = I.bf16_to_f32(p) if bf16 else p
        master[o:o + sizes[k]] = torch.from_numpy(vals.ravel()).to(dev)
    shadow.copy_(master.to(shadow.dtype))
    def views(buf):
        return [buf[int(offs_al[k]):int(offs_al[k]) + sizes[k]].view(shapes[k]) for k in range(len(shapes))]

    pviews, gviews, thviews, vviews = views(shadow), views(gradf), views(master), views(vstate)
    x_np, y_np = I.make_batch(wl, seed=0 if vocab_par else rank, step=1)   # vocabulary ranks share the batch
    x_host = torch.from_numpy(x_np.view(np.int16) if bf16 else x_np).pin_memory()
    y_host = torch.from_numpy(y_np).pin_memory()
    x_dev = (x_host.to(dev).view(torch.bfloat16) if bf16 else x_host.to(dev))
    y_dev = y_host.to(dev)
    q = torch.zeros(wl_model.vocab, dtype=torch.float32, device=dev)
    model = B.BomModel(B.config_for(wl_model, LAM, B1))
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)   # 256 MiB > L2
    gt = B.BOM_BF16 if bf16 else B.BOM_F32
    N = wl.n_rows

    # the sharded steps update after their exchanges: a separate update pass
    fused = not a.separate_update and not dp and not vocab_par
    if fused:   # BOM-AdamW applied inside bom_step, in the epilogues of the weight-gradient GEMMs
        B.bom_set_fused_update(model.h, thviews, vviews, I.weight_decay_mask(wl, WD), LR, B2, EPS)
    xch = torch.zeros(wl.vocab + 3, dtype=torch.float64, device=dev)

    def allreduce(tensor):   # on the step's stream (torch's current stream)
        if dist is not None:
            dist.all_reduce(tensor)

    if vocab_par:
        lse_part = torch.empty(N, dtype=torch.float32, device=dev)
        lse_parts = torch.empty((world, N), dtype=torch.float32, device=dev)
        dh = torch.empty((N, wl.d_model), dtype=torch.float32, device=dev)

    def allgather(out, part):
        if dist is not None:
            dist.all_gather(list(out.unbind(0)), part)
        else:
            out[0].copy_(part)

    def step(t, xx=x_dev, yy=y_dev):
        if fused:
            model.step(xx, yy, N, pviews, q, t, None, None, stream)
        elif dp:
            dp_step(B, model.h, xx, yy, N, pviews, q, t, xch, gviews, gradf, allreduce, stream)
            B.bom_update(master, gradf, gt, None, vstate, shadow if bf16 else None, P, LR, WD, LAM, B2, EPS, t,
                         stream)
        elif vocab_par:
            vocab_step(B, model.h, xx, yy, N, pviews, V_total, v_first, q, t, lse_part, lse_parts, dh, gviews,
                       allgather, allreduce, stream)
            B.bom_update(master, gradf, gt, None, vstate, shadow if bf16 else None, P, LR, WD, LAM, B2, EPS, t,
                         stream)
        else:
            model.step(xx, yy, N, pviews, q, t, gviews, None, stream)
            B.bom_update(master, gradf, gt, None, vstate, shadow if bf16 else None, P, LR, WD, LAM, B2, EPS, t,
                         stream)

    t = 0
    loss_first = None
    for _ in range(a.warmup):
        t += 1
        step(t)
        if t == 1:
            loss_first = model.stats(stream)["loss"]
    model.stats(stream)   # sync + raises if the device latched an error

    # ---------------------------------------------------------------- timed region
    props = torch.cuda.get_device_properties(dev)
    if all(hasattr(props, f) for f in ("pci_domain_id", "pci_bus_id", "pci_device_id")):
        gpu_id = f"{props.pci_domain_id:08X}:{props.pci_bus_id:02X}:{props.pci_device_id:02X}.0"
    else:
        gpu_id = local
    clocks = ClockSampler(gpu_id)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(a.steps)]
    launches0 = B.bom_launch_count()
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    clocks.mark_start()
    # the headline: untraced steps (an event pair around every launch would
    # break the programmatic-dependent-launch overlap of consecutive kernels),
    # one event pair per step, the L2 flush outside it, no host sync between
    for i in range(a.steps):
        flush.zero_()
        t += 1
        ev[i][0].record(stream)
        step(t)
        ev[i][1].record(stream)
    torch.cuda.synchronize()
    clocks.mark_end()
    clk = clocks.stop()
    launches = B.bom_launch_count() - launches0
    st = model.stats(stream)
    step_ms = [e0.elapsed_time(e1) for e0, e1 in ev]
    tot_ms = _max_over_ranks(dist, sum(step_ms), dev)
    # tokens the whole job processes per step: every rank's rows, except under
    # vocabulary parallelism, where all ranks work on the same rows
    job_rows = N if vocab_par else world * N
    value = job_rows * a.steps / (tot_ms / 1e3)

    # the per-kernel split: separate steps with an event pair around every
    # launch (the device time of each kernel class and its algorithmic work)
    per_kernel = {}
    n_traced = max(3, a.steps // 2)
    B.bom_trace(model.h, True)
    for i in range(n_traced):
        flush.zero_()
        t += 1
        step(t)
        for name, fl, by, ms in B.bom_trace_read(model.h, stream):
            d = per_kernel.setdefault(name, [0.0, 0.0, 0.0, 0])
            d[0] += fl
            d[1] += by
            d[2] += ms
            d[3] += 1
    B.bom_trace(model.h, False)
    model.stats(stream)
    traced_ms = sum(v[2] for v in per_kernel.values()) / n_traced

    # ---------------------------------------------------------------- dominant kernel roofline
    dom = max(per_kernel.items(), key=lambda kv: kv[1][2])
    total_dev = sum(v[2] for v in per_kernel.values())
    name, (fl, by, ms, cnt) = dom
    if fl > 0:
        achieved = fl / (ms / 1e3) / 1e12
        roof = {"bound": "tensor", "kernel": name, "achieved": achieved, "peak": peaks["bf16_tflops_sustained"],
                "unit": "TFLOP/s", "frac": achieved / peaks["bf16_tflops_sustained"],
                "peak_source": f"{peak_src} (sustained bf16; kernel timed inside a long step)",
                "frac_of_burst_peak": achieved / peaks["bf16_tflops"],
                "flops_per_launch": fl / cnt, "launches": cnt, "avg_launch_ms": ms / cnt,
                "share_of_device_time": ms / total_dev}
        if name == "gemm_tc.update.mm":
            roof["note"] = ("weight-gradient GEMMs whose epilogue also applies the BOM-AdamW update of each weight "
                            "(18 B/element of theta, v and the bf16 copy); the time includes that update")
    else:
        achieved = by / (ms / 1e3) / 1e9
        roof = {"bound": "hbm", "kernel": name, "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": achieved / peaks["hbm_gbs"], "peak_source": peak_src, "bytes_per_launch": by / cnt,
                "launches": cnt, "avg_launch_ms": ms / cnt, "share_of_device_time": ms / total_dev}
    # GEMM engine as a whole (all tcgen05 launches of the step)
    gem = [v for k, v in per_kernel.items() if k.startswith("gemm_tc")]
    if gem:
        gfl = sum(v[0] for v in gem)
        gms = sum(v[2] for v in gem)
        roof["all_gemm_tflops"] = gfl / (gms / 1e3) / 1e12
        roof["all_gemm_frac"] = roof["all_gemm_tflops"] / peaks["bf16_tflops_sustained"]
        roof["all_gemm_share_of_device_time"] = gms / total_dev
    roof["traffic"] = _ncu_traffic(name)

    kernels = {k: {"ms_per_step": v[2] / n_traced, "launches_per_step": v[3] / n_traced,
                   "tflops": (v[0] / (v[2] / 1e3) / 1e12) if v[0] else None,
                   "gbs": v[1] / (v[2] / 1e3) / 1e9} for k, v in sorted(per_kernel.items(), key=lambda kv: -kv[1][2])}

    # ---------------------------------------------------------------- end to end through host buffers
    # Every step copies its inputs from pinned host memory and reads its
    # statistics (loss, N_t, status) back into pinned host memory.  The copy
    # of step i+1's inputs runs on a second stream into the other of two
    # device buffers while step i computes (a step waits for its own copy, a
    # copy for the step that last used its buffer), and step i's statistics
    # are read and checked on the host while step i+1 runs; the last step's
    # before the clock stops.
    e2e_steps = max(3, a.steps)
    h2d = x_host.numel() * x_host.element_size() + y_host.numel() * y_host.element_size()
    copy_stream = torch.cuda.Stream(device=dev)
    xb = [torch.empty_like(x_host, device=dev) for _ in range(2)]
    yb = [torch.empty_like(y_host, device=dev) for _ in range(2)]
    copied = [torch.cuda.Event() for _ in range(2)]
    freed = [torch.cuda.Event() for _ in range(2)]
    for e in freed:
        e.record(stream)
    sbuf = [torch.empty(B.bom_stats_transfer_bytes(), dtype=torch.uint8).pin_memory() for _ in range(2)]
    sdone = [torch.cuda.Event() for _ in range(2)]

    def issue_copy(j):
        with torch.cuda.stream(copy_stream):
            copy_stream.wait_event(freed[j % 2])
            xb[j % 2].copy_(x_host, non_blocking=True)
            yb[j % 2].copy_(y_host, non_blocking=True)
            copied[j % 2].record(copy_stream)

    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    issue_copy(0)
    for i in range(e2e_steps):
        t += 1
        if i + 1 < e2e_steps:
            issue_copy(i + 1)
        stream.wait_event(copied[i % 2])
        xx = xb[i % 2]
        step(t, xx.view(torch.bfloat16) if bf16 else xx, yb[i % 2])
        freed[i % 2].record(stream)
        B.bom_get_stats_async(model.h, sbuf[i % 2], stream)   # device -> host read of the step's statistics
        sdone[i % 2].record(stream)
        if i > 0:
            sdone[(i - 1) % 2].synchronize()
            B.bom_stats_decode(sbuf[(i - 1) % 2])   # raises if that step latched an error
    sdone[(e2e_steps - 1) % 2].synchronize()
    B.bom_stats_decode(sbuf[(e2e_steps - 1) % 2])
    e2e_s = _max_over_ranks(dist, time.perf_counter() - t0, dev)
    e2e = {"value": job_rows * e2e_steps / e2e_s, "unit": "tokens/s", "h2d_bytes_per_step": int(h2d),
           "d2h_bytes_per_step": B.bom_stats_transfer_bytes()}

    # ---------------------------------------------------------------- sub-measurements
    extra = {}
    if not a.no_extra and rank == 0:
        extra["lm_head_bf16"] = _head_only(B, torch, dev, stream, a, peaks)
        extra["update_sweep"] = _update_sweep(B, torch, dev, stream, a, peaks)
        extra["update_adam_mini_lm_block"] = _adam_mini_only(B, torch, dev, stream, a, peaks)
        extra["update_clipped_lm_block"] = _clipped_update(B, torch, dev, stream, a, peaks)
        extra["telemetry_step_lm_block"] = _telemetry_step(B, torch, dev, stream, a, peaks)
        extra["rmsnorm_lm_block"] = _rmsnorm_step(B, torch, dev, stream, a, peaks)
        extra["small_steps_graph"] = _small_steps(B, torch, dev, stream, a)

    # The two targets of the method's measurement, under keys of the roofline
    # object: the fused head + reprojection step (LM output block) against the
    # bf16 tensor peak, and the update alone against the HBM copy peak.
    roof["timing"] = ("headline from untraced steps; kernel times from separate steps with an event pair "
                      "around every launch")
    roof["traced_step_ms"] = traced_ms
    if "lm_head_bf16" in extra:
        hd = extra["lm_head_bf16"]
        roof["head_step_tokens_per_s"] = hd["value"]
        roof["head_step_ms"] = hd["ms_per_step"]
        roof["head_step_frac_of_bf16_peak"] = hd["step_frac_of_bf16_peak"]
    for size, u in extra.get("update_sweep", {}).items():
        roof[f"update_gbs_{size}"] = u["value"]
        roof[f"update_frac_of_hbm_{size}"] = u["frac_of_hbm"]

    cpu = None
    if rank == 0 and world == 1 and not a.no_cpu:
        v, desc, _ = oracle_sample(wl)
        cpu = {"value": v, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle", "sample": desc}

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": a.steps,
                "warmup": a.warmup, "ms_per_step": tot_ms / a.steps, "higher_is_better": True,
                "scaling": "strong" if vocab_par else "weak",
                "vs_baseline": None, "dtype": "bf16" if bf16 else "f32",
                "data": "synthetic: seeded N(0,1) inputs, Kaiming-uniform MLP weights, N(0,0.02) head, "
                        "Zipf(1.1) labels",
                "config": {"workload": _workload_desc(wl), "global_batch": job_rows, "tokens_per_gpu": N,
                           "parallelism": (f"dp{world}: rows split across ranks, all-reduce of the V + 3 exchange "
                                           "sums and of the bf16 gradient shares, separate update; measured on "
                                           "one GPU only" if dp else
                                           f"vocab{world}: head columns split across ranks, every rank with the "
                                           "whole batch, all-gather of the row log-sum-exp parts and all-reduce "
                                           "of the head's input cotangent, separate update; not measured on "
                                           "hardware" if vocab_par else f"replicas x{world} (no data-path collective)"),
                           "l2": "flushed between timed steps (256 MiB write outside the step events)",
                           "lr": LR, "weight_decay": WD, "lambda": LAM, "beta1": B1, "beta2": B2,
                           "update": "fused into the weight-gradient GEMM epilogues" if fused else "separate pass",
                           "step": ("bom_step_shard_begin, all-reduce, bom_step_shard_end, all-reduce, bom_update"
                                    if dp else "bom_step_vshard_begin, all-gather, bom_step_vshard_mid, all-reduce, "
                                    "bom_step_vshard_end, bom_update" if vocab_par else
                                    "bom_step" + ("" if fused else ", bom_update"))},
                "roofline": roof, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": int(launches),
                "clocks": clk, "loss_first_step": loss_first, "loss": st["loss"], "kernels": kernels,
                "sub": extra}
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()


def dp_step(lib, h, x, y, n_rows, params, q, t, xch, grads, grad_flat, allreduce, stream=None):
    """One data-parallel BOM step of this rank's rows.  Algorithm 1's s_t and
    the surrogate's 1/N_t are means over the supervised rows of the whole
    batch, so the step splits at one exchange: this rank's part up to the
    column sums of its residuals (bom_step_shard_begin writes them, its CE sum,
    its N_t and an error flag into xch, V + 3 doubles), the sum of every rank's
    xch, the rest of the step with the whole batch's N_t, s_t and qhat_t
    (bom_step_shard_end writes this rank's share of u into grads, views of
    grad_flat), then the sum of the ranks' shares.  `allreduce(t)` sums a
    tensor over the ranks in place (nothing on one rank); `lib` is the
    binding module."""
    lib.bom_step_shard_begin(h, x, y, n_rows, params, xch, stream)
    allreduce(xch)
    lib.bom_step_shard_end(h, x, y, n_rows, params, q, t, xch, grads, None, stream)
    allreduce(grad_flat)


def vocab_step(lib, h, x, y, n_rows, params, v_total, v_first, q, t, lse_part, lse_parts, dh, grads, allgather,
               allreduce, stream=None):
    """One vocabulary-parallel BOM step: this rank holds rows v_first.. of the
    head (and the same rows of q), the whole backbone and the whole batch.  A
    row's residual needs the other ranks' columns only through its
    log-sum-exp (Algorithm 1), and the head's input cotangent is a sum over
    columns (Eq. mix-gradient): this rank's part of each row's log-sum-exp
    (bom_step_vshard_begin), the parts of every rank gathered in rank order
    into lse_parts, the residuals, s_t, q_t and the head rows of u of this
    rank's columns with its part of the cotangent (bom_step_vshard_mid), the
    sum of the parts, and the backbone's backward from it
    (bom_step_vshard_end), whose u is the same on every rank.
    `allgather(out, part)` fills out[r] with rank r's part, `allreduce(t)`
    sums a tensor over the ranks in place; `lib` is the binding module."""
    lib.bom_step_vshard_begin(h, x, y, n_rows, params, v_total, v_first, lse_part, stream)
    allgather(lse_parts, lse_part)
    lib.bom_step_vshard_mid(h, x, y, n_rows, params, q, t, lse_parts, lse_parts.shape[0], grads, dh, stream)
    allreduce(dh)
    lib.bom_step_vshard_end(h, x, y, n_rows, params, dh, grads, stream)


def _max_over_ranks(dist, x, dev):
    """The largest of a per-rank time over all ranks (x itself on one rank),
    so a whole-job rate is set by the slowest replica."""
    if dist is None:
        return x
    import torch
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def _ncu_traffic(kernel_name):
    """DRAM bytes per launch of `kernel_name` from the committed ncu summary,
    valid only while the kernel source is unchanged since the capture."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    if not os.path.exists(path):
        return None
    try:
        import hashlib
        d = json.load(open(path))
        rec = d.get(kernel_name)
        if not rec:
            return None
        src = open(os.path.join(ROOT, rec["source"]), "rb").read()
        if hashlib.sha256(src).hexdigest() != rec["sha256"]:
            return None
        return rec["dram_bytes_per_launch"]
    except Exception:
        return None


def _head_only(B, torch, dev, stream, a, peaks):
    """LM output block alone: 8192 tokens x d 768, vocab 50257 (forward logits,
    CE statistics, residuals, s/q, head dW and dH with the reprojection)."""
    wl = I.LM_HEAD_BF16
    params = [torch.from_numpy(p.view(np.int16)).to(dev).view(torch.bfloat16) for p in I.init_params(wl, 0)]
    x_np, y_np = I.make_batch(wl, 0, 1)
    x = torch.from_numpy(x_np.view(np.int16)).to(dev).view(torch.bfloat16)
    y = torch.from_numpy(y_np).to(dev)
    grads = [torch.empty_like(p) for p in params]
    dx = torch.empty_like(x)
    q = torch.zeros(wl.vocab, dtype=torch.float32, device=dev)
    m = B.BomModel(B.config_for(wl))
    B.bom_set_input_grad(m.h, dx)
    for t in range(1, a.warmup + 1):
        m.step(x, y, wl.n_rows, params, q, t, grads, None, stream)
    m.stats(stream)
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)
    # the step time: no trace events between the kernels (they would break the
    # programmatic-dependent-launch overlap of consecutive kernels)
    tot = 0.0
    t = a.warmup
    for i in range(a.steps):
        flush.zero_()
        t += 1
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        m.step(x, y, wl.n_rows, params, q, t, grads, None, stream)
        e1.record(stream)
        torch.cuda.synchronize()
        tot += e0.elapsed_time(e1)
    # the per-kernel split: separate steps with an event pair around every launch
    B.bom_trace(m.h, True)
    gem_fl = gem_ms = 0.0
    per = {}
    n_tr = max(3, a.steps // 4)
    for i in range(n_tr):
        flush.zero_()
        t += 1
        m.step(x, y, wl.n_rows, params, q, t, grads, None, stream)
        for name, fl, by, ms in B.bom_trace_read(m.h, stream):
            per[name] = per.get(name, 0.0) + ms / n_tr
            if name.startswith("gemm_tc"):
                gem_fl += fl
                gem_ms += ms
    B.bom_trace(m.h, False)
    m.stats(stream)
    m.close()
    flops = 3 * 2.0 * wl.n_rows * wl.d_in * wl.vocab
    return {"workload": "LM output block: H 8192x768, head 50257x768 (tied-head shape), Zipf(1.1) labels; "
                        "logits + CE, residuals, s_t, q_t, head dW and dH with the reprojection",
            "value": wl.n_rows * a.steps / (tot / 1e3), "unit": "tokens/s", "ms_per_step": tot / a.steps,
            "step_tflops": flops / (tot / a.steps / 1e3) / 1e12,
            "step_frac_of_bf16_peak": flops / (tot / a.steps / 1e3) / 1e12 / peaks["bf16_tflops"],
            "gemm_tflops": gem_fl / (gem_ms / 1e3) / 1e12 if gem_ms else None,
            "kernels_ms_per_step": {k: round(v, 4) for k, v in sorted(per.items(), key=lambda kv: -kv[1])},
            "timing": "step time from untraced steps; per-kernel split from separate steps traced with an event "
                      "pair around every launch"}


def _update_sweep(B, torch, dev, stream, a, peaks):
    """BOM-AdamW update alone over flat buffers of 10M, 125M and 1e9 elements
    (fp32 theta / h / v, bf16 g; 22 B/element), L2 flushed before each run."""
    out = {}
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)
    for n in I.UPDATE_SIZES:
        theta, g, h, v = I.update_sweep_device(n, 0, dev)
        for t in range(1, 4):
            B.bom_update(theta, g, B.BOM_BF16, h, v, None, n, LR, 0.01, LAM, B2, EPS, t, stream)

        def run(i):
            B.bom_update(theta, g, B.BOM_BF16, h, v, None, n, LR, 0.01, LAM, B2, EPS, 4 + i, stream)

        med = _timed(torch, stream, run, max(5, a.steps // 2), flush)
        gbs = 22.0 * n / (med / 1e3) / 1e9
        del theta, g, h, v
        torch.cuda.empty_cache()
        out[f"{n:.3g}".replace("+0", "").replace("+", "")] = {
            "workload": f"update sweep, {n} elements: read theta f32, g bf16, h f32, v f32; write theta, v "
                        "(22 B/element)", "value": gbs, "unit": "GB/s", "ms": med,
            "frac_of_hbm": gbs / peaks["hbm_gbs"], "peak_source": "measured copy bandwidth"}
    return out


def _small_steps(B, torch, dev, stream, a):
    """The two small configurations (tiny fp32 MLP classifier, batch 32; vision
    head, 3-layer bf16 MLP at batch 256, 1000 classes), BOM step with the fused
    update: launched kernel by kernel, and as one captured step (CUDA graph)
    that reads t and lr from the device.  Steps run back to back (a few MB,
    L2-resident), so the time includes what launching costs; each timing
    starts a second after the previous GPU work."""
    out = {}
    for wl in (I.TINY_MLP_F32, I.VISION_HEAD_BF16):
        bf16 = wl.dtype == "bf16"
        res = {}
        for mode in ("launches", "graph"):
            params_np = I.init_params(wl, 0)
            if bf16:
                params = [torch.from_numpy(p.view(np.int16)).to(dev).view(torch.bfloat16) for p in params_np]
                theta = [torch.from_numpy(I.bf16_to_f32(p)).to(dev) for p in params_np]
            else:
                params = [torch.from_numpy(p.copy()).to(dev) for p in params_np]
                theta = [torch.from_numpy(p.copy()).to(dev) for p in params_np]
            v = [torch.zeros(p.shape, dtype=torch.float32, device=dev) for p in params_np]
            x_np, y_np = I.make_batch(wl, 0, 1)
            x = (torch.from_numpy(x_np.view(np.int16)).to(dev).view(torch.bfloat16) if bf16
                 else torch.from_numpy(x_np).to(dev))
            y = torch.from_numpy(y_np).to(dev)
            q = torch.zeros(wl.vocab, dtype=torch.float32, device=dev)
            m = B.BomModel(B.config_for(wl, LAM, B1))
            B.bom_set_fused_update(m.h, theta, v, I.weight_decay_mask(wl, WD), LR, B2, EPS)
            g = None
            if mode == "graph":
                t_dev = torch.ones(1, dtype=torch.int64, device=dev)
                B.bom_set_step_scalars(m.h, t_dev, None)
                g = B.bom_graph_capture(m.h, x, y, wl.n_rows, params, q, None, None)
                run = lambda t: B.bom_graph_launch(g, stream)
            else:
                run = lambda t: m.step(x, y, wl.n_rows, params, q, t, None, None, stream)
            # a second without GPU work first: the power cap is a running
            # average, so this light workload then runs at the SM clock it
            # holds on its own, not at the one the preceding (power-capped)
            # measurements left
            torch.cuda.synchronize()
            time.sleep(1.0)
            t = 0
            for _ in range(a.warmup):
                t += 1
                run(t)
            m.stats(stream)
            K = 200
            n0 = B.bom_launch_count()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for t in range(t + 1, t + 1 + K):
                run(t)
            e1.record(stream)
            torch.cuda.synchronize()
            ms = e0.elapsed_time(e1) / K
            kpl = (B.bom_launch_count() - n0) / K
            m.stats(stream)
            res[mode] = {"value": wl.n_rows / (ms / 1e3), "unit": "tokens/s", "us_per_step": 1e3 * ms,
                         "kernels_per_step": kpl}
            if g is not None:
                B.bom_graph_destroy(g)
            m.close()
        res["workload"] = _workload_desc(wl)
        res["graph_speedup"] = res["launches"]["us_per_step"] / res["graph"]["us_per_step"]
        out[wl.name] = res
    return out


def _lm_state(B, torch, dev, wl, seed=0):
    """Device parameters (bf16), fp32 masters, a batch and q for workload wl."""
    params_np = I.init_params(wl, seed)
    params = [torch.from_numpy(p.view(np.int16)).to(dev).view(torch.bfloat16) for p in params_np]
    theta = [torch.from_numpy(I.bf16_to_f32(p)).to(dev) for p in params_np]
    x_np, y_np = I.make_batch(wl, seed, 1)
    x = torch.from_numpy(x_np.view(np.int16)).to(dev).view(torch.bfloat16)
    y = torch.from_numpy(y_np).to(dev)
    q = torch.zeros(wl.vocab, dtype=torch.float32, device=dev)
    return params, theta, x, y, q


def _timed(torch, stream, fn, n_iter, flush):
    """Median CUDA-event time (ms) of fn() over n_iter runs, L2 flushed before each."""
    ms = []
    for i in range(n_iter):
        flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        fn(i)
        e1.record(stream)
        torch.cuda.synchronize()
        ms.append(e0.elapsed_time(e1))
    return statistics.median(ms)


def _clipped_update(B, torch, dev, stream, a, peaks):
    """Global-norm clipping of u over the LM block's 166,199,296 parameters:
    the fixed-order sum of u^2 (bf16 u) and the clipped BOM-AdamW update."""
    wl = I.LM_MLP_BF16
    P = wl.n_params()
    gen = torch.Generator(device=dev)
    gen.manual_seed(1)
    theta = torch.randn(P, generator=gen, device=dev) * 1e-2
    u = (torch.randn(P, generator=gen, device=dev) * 1e-3).to(torch.bfloat16)
    v = torch.zeros(P, dtype=torch.float32, device=dev)
    shadow = torch.empty(P, dtype=torch.bfloat16, device=dev)
    sq = torch.zeros(1, dtype=torch.float64, device=dev)
    m = B.BomModel(B.config_for(I.TINY_MLP_F32))   # a handle for the partials buffer
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)

    def run(i):
        sq.zero_()
        B.bom_sqnorm(m.h, u, B.BOM_BF16, None, LAM, P, sq, stream)
        B.bom_update_clipped(theta, u, B.BOM_BF16, None, v, shadow, P, LR, WD, LAM, B2, EPS, 4 + i, sq, 1.0, stream)

    for i in range(3):
        run(i)
    ms = _timed(torch, stream, run, max(5, a.steps // 2), flush)
    m.close()
    gbs = 22.0 * P / (ms / 1e3) / 1e9
    del theta, u, v, shadow
    torch.cuda.empty_cache()
    return {"workload": "global-norm clipping (max norm 1.0) of bf16 u over 166,199,296 parameters: sum of u^2 "
                        "(2 B/element) + clipped update (read theta, u, v; write theta, v, bf16 copy: 20 B/element)",
            "value": gbs, "unit": "GB/s", "ms": ms, "frac_of_hbm": gbs / peaks["hbm_gbs"],
            "peak_source": "measured copy bandwidth"}


def _telemetry_step(B, torch, dev, stream, a, peaks):
    """Own-step control with drift telemetry on the LM block (16384 tokens):
    one bom_step in G_AND_H mode with an own-step output (backward passes for
    g, h = Jbar^T qhat and o = Jbar^T s_t, residual norms), then the own-step
    moment with the drift sums of head and encoder over all parameters."""
    wl = I.LM_MLP_BF16
    params, theta, x, y, q = _lm_state(B, torch, dev, wl)
    f32 = torch.float32
    grads = [torch.empty_like(p) for p in params]
    hs = [torch.empty(p.shape, dtype=f32, device=dev) for p in params]
    os_ = [torch.empty(p.shape, dtype=f32, device=dev) for p in params]
    Ms = [torch.zeros(p.shape, dtype=f32, device=dev) for p in params]
    mh = [torch.empty(p.shape, dtype=f32, device=dev) for p in params]
    sums = torch.zeros((2, 4), dtype=torch.float64, device=dev)
    m = B.BomModel(B.config_for(wl, LAM, B1, B.BOM_OUT_G_AND_H))
    B.bom_set_own_step_output(m.h, os_)
    head = len(params) - 1
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)
    per = {}

    def moments(t):
        sums.zero_()
        for k in range(len(params)):
            B.bom_own_step_moment(m.h, Ms[k], os_[k], hs[k], mh[k], Ms[k].numel(), B1, t,
                                  sums[0] if k == head else sums[1], stream)

    def run(i):
        t = 1 + i
        m.step(x, y, wl.n_rows, params, q, t, grads, hs, stream)
        moments(t)

    for i in range(2):
        run(i)
    B.bom_trace(m.h, True)
    ms = _timed(torch, stream, lambda i: run(3 + i), max(3, a.steps // 4), flush)
    for name, fl, by, kms in B.bom_trace_read(m.h, stream):
        per[name] = per.get(name, 0.0) + kms
    mom_ms = _timed(torch, stream, lambda i: moments(20 + i), 3, flush)
    st = m.stats(stream)
    s_ = sums.cpu().numpy()
    P = wl.n_params()
    m.close()
    del grads, hs, os_, Ms, mh, params, theta
    torch.cuda.empty_cache()
    return {"workload": "LM block + 2 SwiGLU MLPs, 16384 tokens: own-step control step with drift telemetry "
                        "(forward, task space, three backward passes g / h / own-step, residual norms, "
                        "M_t and the drift sums over 166,199,296 parameters)",
            "value": wl.n_rows / (ms / 1e3), "unit": "tokens/s", "ms_per_step": ms,
            "cancel_ratio": st["cancel"],
            "drift_cos_head": float(s_[0, 0] / np.sqrt(s_[0, 1] * s_[0, 2])),
            "drift_cos_encoder": float(s_[1, 0] / np.sqrt(s_[1, 1] * s_[1, 2])),
            "moment_pass_ms": mom_ms, "moment_pass_gbs": 20.0 * P / (mom_ms / 1e3) / 1e9,
            "kernels_ms_last_step": {k: round(v, 4) for k, v in sorted(per.items(), key=lambda kv: -kv[1])}}


def _rmsnorm_step(B, torch, dev, stream, a, peaks):
    """The LM block with a final RMSNorm before the head (16384 tokens, the
    update fused), against the same step without the norm."""
    wl = I.LM_NORM_BF16
    params, theta, x, y, q = _lm_state(B, torch, dev, wl)
    v = [torch.zeros_like(t) for t in theta]
    m = B.BomModel(B.config_for(wl, LAM, B1))
    B.bom_set_fused_update(m.h, theta, v, I.weight_decay_mask(wl, WD), LR, B2, EPS)
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)

    def run(i):
        m.step(x, y, wl.n_rows, params, q, 1 + i, None, None, stream)

    for i in range(3):
        run(i)
    B.bom_trace(m.h, True)
    ms = _timed(torch, stream, lambda i: run(4 + i), max(3, a.steps // 4), flush)
    per = {}
    for name, fl, by, kms in B.bom_trace_read(m.h, stream):
        if name.startswith("rmsnorm") or name == "colsum":
            d = per.setdefault(name, [0.0, 0.0])
            d[0] += by
            d[1] += kms
    m.stats(stream)
    m.close()
    del params, theta, v
    torch.cuda.empty_cache()
    return {"workload": "LM block + 2 SwiGLU MLPs + final RMSNorm (gamma, weight decay 0), 16384 tokens, "
                        "BOM step with the fused update",
            "value": wl.n_rows / (ms / 1e3), "unit": "tokens/s", "ms_per_step": ms,
            "norm_kernels": {k: {"ms": round(v[1], 4), "gbs": v[0] / (v[1] / 1e3) / 1e9} for k, v in per.items()}}


def _adam_mini_only(B, torch, dev, stream, a, peaks):
    """BOM-Adam-mini update of the LM block's 166,199,296 parameters with one
    second moment per output neuron (row) of every weight matrix, u given in
    bf16 (the numerator bom_step produces), bf16 copy of theta written."""
    wl = I.LM_MLP_BF16
    shapes = [s for _, s, _ in wl.param_shapes()]
    gen = torch.Generator(device=dev)
    gen.manual_seed(0)
    ts = []
    for rows, cols in shapes:
        n = rows * cols
        th = torch.randn(n, generator=gen, device=dev) * 1e-3
        g = (torch.randn(n, generator=gen, device=dev) * 1e-3).to(torch.bfloat16)
        vb = torch.zeros(rows, dtype=torch.float32, device=dev)
        sh = torch.empty(n, dtype=torch.bfloat16, device=dev)
        ts.append((th, g, vb, sh, n, cols))
    P = sum(t[4] for t in ts)
    nblocks = sum(t[2].numel() for t in ts)

    def upd(t):
        for th, g, vb, sh, n, cols in ts:
            B.bom_update_blockshared(th, g, B.BOM_BF16, None, vb, sh, n, cols, LR, WD, LAM, B2, EPS, t, stream)

    for t in range(1, 4):
        upd(t)
    torch.cuda.synchronize()
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)
    ms = []
    for i in range(max(5, a.steps // 2)):
        flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        upd(4 + i)
        e1.record(stream)
        torch.cuda.synchronize()
        ms.append(e0.elapsed_time(e1))
    med = statistics.median(ms)
    gbs = 12.0 * P / (med / 1e3) / 1e9
    del ts
    torch.cuda.empty_cache()
    return {"workload": "BOM-Adam-mini update of the LM block (7 tensors, 166,199,296 parameters), one second "
                        "moment per output neuron: read theta f32, u bf16; write theta f32, bf16 copy "
                        "(12 B/element; each block read once into registers when it has at most 8192 elements)",
            "value": gbs, "unit": "GB/s", "ms": med, "frac_of_hbm": gbs / peaks["hbm_gbs"],
            "second_moment_entries": nblocks, "params": P,
            "state_reduction_vs_elementwise": 1.0 - nblocks / P, "peak_source": "measured copy bandwidth"}


if __name__ == "__main__":
    main()
