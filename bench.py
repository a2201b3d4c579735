#!/usr/bin/env python
"""Benchmark of the SPADE verify step on GB300.

One step = one pass of the whole hot path over one batch of synthetic input:
verify attention (one layer) -> LM head + accept/reject + residual sampling ->
KV commit, all on one stream through the C-ABI library.  The metric is the
number of committed tokens (sum over sequences of accepted drafts + 1) per
second of device time, with inputs resident in HBM.  `e2e` repeats it through
the same public calls with the per-step inputs in pinned host memory, copied
in and the step's result read back inside the timed region.

Default workload: the Llama-3-8B-shaped verifier step (batch 8, GQA 32/8,
head_dim 128, hidden 4096, vocab 128256, ctx 4096, k = 8, stochastic), the
paper's own verifier shape; the other workloads of the suite are timed on the
device after it (`per_workload`).  `--impl reference` times the float64 CPU
oracle on the same workload instead (bounded samples: one sequence per step).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import signal
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import torch  # noqa: E402

from paper_2608_13076_gb300 import workloads as W  # noqa: E402

L2_BYTES = 129 * 1024 * 1024
METRIC = "verified tokens/s per verify step (1 GB300); verify-attn HBM GB/s vs peak"
UNIT = "tokens/s"


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), float(d["bf16_tflops_sustained"]), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


def _traffic(kernel, workload):
    """ncu DRAM bytes per launch for this kernel and workload, if its sources are unchanged."""
    import hashlib
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            rec = json.load(f)[kernel][workload]
        h = hashlib.sha256()
        for src in rec["sources"]:  # every file the kernel is built from, in this order
            with open(os.path.join(ROOT, src), "rb") as f:
                h.update(f.read())
        if h.hexdigest()[:16] != rec["sha256_16"]:
            return None
        return rec["bytes"]
    except Exception:
        return None


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def _job_rate(tokens_local, t_local, ws, device):
    """Whole-job rate of ws replicas: every rank's tokens over the slowest rank's time.

    Returns (rate, slowest time).  With ws > 1 every rank must call it (two
    all-reduces on the default process group).
    """
    if ws > 1:
        t = torch.tensor([t_local], dtype=torch.float64, device=device)
        n = torch.tensor([float(tokens_local)], dtype=torch.float64, device=device)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        torch.distributed.all_reduce(n, op=torch.distributed.ReduceOp.SUM)
        return float(n.item()) / float(t.item()), float(t.item())
    return tokens_local / t_local, t_local


def _head_start(iterations):
    """Queues a spin kernel so that the host can enqueue the timed launches ahead of the
    GPU: a timed region must not contain GPU idle time spent waiting for Python to issue
    the next launch.  It gives the host 0.5 ms per loop iteration (at least 3 ms), far
    above what an iteration takes (tens of microseconds), so a slow or busy host cannot
    leak into a kernel's time."""
    ms = max(3.0, 0.5 * iterations)
    torch.cuda._sleep(int(ms * 2.0e6))  # cycles at about 2 GHz


def _to_device(wl, dev):
    return {k: (v.to(dev) if isinstance(v, torch.Tensor) else v) for k, v in wl.items()}


def _config(spec, wl, ws):
    """The workload's config block, identical for both arms of the benchmark."""
    attn_bytes, lm_bytes, _, _, _ = _work_bytes(wl)
    work_set = attn_bytes + lm_bytes
    return {"workload": spec.name, "B": wl["B"], "Hq": wl["Hq"], "Hkv": wl["Hkv"], "D": wl["D"],
            "H": wl["H"], "V": wl["V"], "ctx": list(spec.ctx), "k": list(spec.k), "mode": spec.mode,
            "rows": wl["R"], "parallelism": "replicas" if ws > 1 else "single",
            "l2": ("flushed between steps" if work_set < 2 * L2_BYTES
                   else f"working set {work_set / 1e9:.2f} GB > L2")}


def _lm_roofline(lm_bytes, lm_flop, t, hbm, bf16_sus, bf16_burst, peak_src):
    """Roofline of the LM-head kernel timed inside a step: the bound is whichever of its
    HBM bytes and its bf16 flops takes longer at peak (sustained bf16 for a kernel in a
    long step); the fraction is taken against that bound's peak."""
    t_hbm = lm_bytes / (hbm * 1e9)
    t_tc = lm_flop / (bf16_sus * 1e12)
    tensor = {"tflops": lm_flop / t / 1e12, "frac_of_sustained": lm_flop / t / 1e12 / bf16_sus,
              "frac_of_burst": lm_flop / t / 1e12 / bf16_burst,
              "ceiling_frac_of_sustained": min(1.0, t_tc / t_hbm) if t_hbm > 0 else 1.0}
    if t_tc > t_hbm:
        r = {"bound": "tensor", "achieved": lm_flop / t / 1e12, "peak": bf16_sus, "unit": "TFLOP/s",
             "frac": lm_flop / t / 1e12 / bf16_sus, "peak_kind": "bf16_tflops_sustained"}
    else:
        r = {"bound": "hbm", "achieved": lm_bytes / t / 1e9, "peak": hbm, "unit": "GB/s",
             "frac": lm_bytes / t / 1e9 / hbm, "peak_kind": "hbm_gbs"}
    r.update({"algorithmic_bytes": lm_bytes, "algorithmic_flop": lm_flop, "peak_source": peak_src,
              "tensor": tensor})
    return r


def _work_bytes(wl):
    """Algorithmic bytes of the two dominant kernels for one step."""
    ctx = wl["ctx_lens"].long().cpu()
    kd = wl["n_draft"].long().cpu()
    keys = int((ctx + kd + 1).sum())
    attn = keys * wl["Hkv"] * wl["D"] * 2 * 2 + 2 * wl["R"] * wl["Hq"] * wl["D"] * 2
    n_stoch = int((wl["mode"].cpu() == W.STOCHASTIC).sum()) if wl["draft_probs"] is not None else 0
    lm = wl["V"] * wl["H"] * 2 + wl["R"] * wl["H"] * 2 + n_stoch * wl["V"] * 4
    lm_flop = 2.0 * wl["R"] * wl["V"] * wl["H"]
    attn_flop = 0.0
    G = wl["Hq"] // wl["Hkv"]
    for b in range(wl["B"]):
        for i in range(int(kd[b]) + 1):
            attn_flop += 4.0 * wl["D"] * (int(ctx[b]) + i + 1) * wl["Hkv"] * G
    return attn, lm, lm_flop, attn_flop, keys


class Clocks:
    """Samples nvidia-smi clocks and throttle reasons while running."""

    def __init__(self, index):
        self.proc = None
        self.path = None
        self.index = index

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index),
                 "--query-gpu=clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                 "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                 "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            time.sleep(0.2)
            self.proc.send_signal(signal.SIGTERM)
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if self.proc is None or not self.path:
            return None
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 8:
                    continue
                try:
                    sm.append(float(parts[0]))
                    mx.append(float(parts[1]))
                except ValueError:
                    continue
                for n, v in zip(names, parts[4:8]):
                    if v.lower() == "active":
                        reasons.add(n)
        os.unlink(self.path)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


# ---------------------------------------------------------------------------
def run_spade(args, ws, rank, local):
    import paper_2608_13076_gb300 as spade
    from paper_2608_13076_gb300 import _build

    if rank == 0 or not _build.up_to_date():
        _build.build()
    if ws > 1:
        torch.distributed.barrier()
    spade.load()
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    spec = W.SPECS[args.workload]
    # Inputs are drawn on the CPU (a seed names the same data on every device);
    # the CPU copy stays untouched for the oracle, the GPU copy is stepped.
    wl_cpu = W.make_workload(spec, device="cpu")
    wl = _to_device(wl_cpu, dev)
    B, R = wl["B"], wl["R"]
    max_k = int(wl["n_draft"].max())
    out = torch.empty_like(wl["q"])
    acc = torch.zeros(B, dtype=torch.int32, device=dev)
    tok = torch.zeros(B, dtype=torch.int32, device=dev)
    status = spade.status_tensor(dev)
    ws_attn = spade.attn_workspace(B, wl["Hq"], wl["Hkv"], wl["D"], wl["cap"], max_k, device=dev)
    ws_acc = spade.accept_workspace(B, R, wl["H"], wl["V"], device=dev)
    ctx0 = wl["ctx_lens"].clone()
    stream = torch.cuda.current_stream()

    def step(inputs, evs=None, outs=None):
        a_out, t_out = outs if outs is not None else (acc, tok)
        if evs:
            evs[0].record(stream)
        spade.spade_verify_attention(inputs["q"], wl["k_cache"], wl["v_cache"], inputs["ctx_lens"],
                                     inputs["n_draft"], inputs["cu_q"], out, None, max_k=max_k,
                                     workspace=ws_attn, status=status)
        if evs:
            evs[1].record(stream)
        if args.separate_commit:
            spade.spade_verify_accept(inputs["hidden"], wl["w_lm"], inputs["draft_tokens"],
                                      inputs["draft_probs"], inputs["uniforms"], inputs["mode"], inputs["cu_q"],
                                      inputs["n_draft"], a_out, t_out, workspace=ws_acc, status=status)
            if evs:
                evs[2].record(stream)
            spade.spade_kv_commit(wl["k_cache"], wl["v_cache"], inputs["ctx_lens"], a_out, inputs["n_draft"],
                                  status=status)
        else:
            # Accept + KV commit in one launch (the commit runs inside the LM-head kernel).
            spade.spade_verify_accept_commit(inputs["hidden"], wl["w_lm"], inputs["draft_tokens"],
                                             inputs["draft_probs"], inputs["uniforms"], inputs["mode"],
                                             inputs["cu_q"], inputs["n_draft"], a_out, t_out, wl["k_cache"],
                                             wl["v_cache"], inputs["ctx_lens"], workspace=ws_acc, status=status)
            if evs:
                evs[2].record(stream)
        if evs:
            evs[3].record(stream)

    attn_bytes, lm_bytes, lm_flop, attn_flop, keys = _work_bytes(wl)
    work_set = attn_bytes + lm_bytes
    flush = work_set < 2 * L2_BYTES
    flush_buf = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device=dev) if flush else None

    for _ in range(args.warmup):
        wl["ctx_lens"].copy_(ctx0)
        step(wl)
    torch.cuda.synchronize()
    if int(status.item()) & ~spade.DEV_FALLBACK:
        raise RuntimeError(f"device status {int(status.item())} after warm-up")
    tokens_per_step = int((acc.long() + 1).sum().item())

    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
    if ws > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with Clocks(local) as clk:
        t_wall0 = time.perf_counter()
        _head_start(args.steps)
        for s in range(args.steps):
            wl["ctx_lens"].copy_(ctx0)
            if flush:
                flush_buf.zero_()
            step(wl, evs[s])
        torch.cuda.synchronize()
        t_wall = time.perf_counter() - t_wall0
    if ws > 1:
        torch.distributed.barrier()
    t_step = [e[0].elapsed_time(e[3]) * 1e-3 for e in evs]
    t_attn = [e[0].elapsed_time(e[1]) * 1e-3 for e in evs]
    t_acc = [e[1].elapsed_time(e[2]) * 1e-3 for e in evs]
    t_com = [e[2].elapsed_time(e[3]) * 1e-3 for e in evs]
    value, total = _job_rate(tokens_per_step * args.steps, sum(t_step), ws, dev)

    # ---- end to end through the public API with pinned host inputs -------------
    # Every step copies its inputs from pinned host memory and reads its result
    # back inside the timed region.  The inputs of step i+1 are copied on a
    # second stream into the other of two device buffers while step i runs
    # (the usual double buffering of a serving loop).
    e2e = None
    if not args.no_e2e:
        host_keys = ["q", "hidden", "draft_tokens", "draft_probs", "uniforms", "mode", "cu_q", "n_draft",
                     "ctx_lens"]
        src = {k: (wl[k] if k != "ctx_lens" else ctx0) for k in host_keys if wl[k] is not None}
        # The step's inputs live in one pinned host arena (256-byte aligned
        # views, as a serving loop's staging buffer would hold them) and move
        # with one copy per step into one of two device arenas.
        offs, off = {}, 0
        for k, t in src.items():
            offs[k] = off
            off += (t.numel() * t.element_size() + 255) // 256 * 256
        arena_bytes = off
        host_arena = torch.empty(arena_bytes, dtype=torch.uint8).pin_memory()

        def carve(arena):
            return {k: arena[offs[k]:offs[k] + t.numel() * t.element_size()].view(t.dtype).view(t.shape)
                    for k, t in src.items()}

        host = carve(host_arena)
        for k, t in src.items():
            host[k].copy_(t.cpu())
        dev_arenas = [torch.empty(arena_bytes, dtype=torch.uint8, device=dev) for _ in range(2)]
        bufs = [carve(a) for a in dev_arenas]
        for bset in bufs:
            bset["draft_probs"] = bset.get("draft_probs")
        # accepted_len and next_token side by side: one read-back per step.
        res_dev = torch.empty(2 * B, dtype=torch.int32, device=dev)
        acc_e2e, tok_e2e = res_dev[:B], res_dev[B:]
        res_host = torch.empty(2 * B, dtype=torch.int32).pin_memory()
        h2d = sum(t.numel() * t.element_size() for t in src.values())
        d2h = res_host.numel() * 4
        n_e2e = max(3, min(args.steps, 100))  # the first step's own copy is the pipeline fill
        copy_stream = torch.cuda.Stream(device=dev)
        copied = [torch.cuda.Event() for _ in range(2)]
        consumed = [torch.cuda.Event() for _ in range(2)]
        e_start = torch.cuda.Event(enable_timing=True)
        e_end = torch.cuda.Event(enable_timing=True)

        def issue_copy(i):
            with torch.cuda.stream(copy_stream):
                if i >= 2:
                    copy_stream.wait_event(consumed[i % 2])  # step i-2 is done with this buffer
                dev_arenas[i % 2].copy_(host_arena, non_blocking=True)
                copied[i % 2].record(copy_stream)

        total_it = n_e2e + 2
        torch.cuda.synchronize()
        for it in range(total_it):
            if it == 0:
                issue_copy(0)
            if it == 2:  # two untimed steps first; the timed region starts with step 2's own copy
                torch.cuda.synchronize()
                e_start.record(stream)
                copy_stream.wait_event(e_start)
                issue_copy(2)
            stream.wait_event(copied[it % 2])
            step(bufs[it % 2], outs=(acc_e2e, tok_e2e))
            consumed[it % 2].record(stream)
            res_host.copy_(res_dev, non_blocking=True)
            if it + 1 < total_it and it + 1 != 2:
                issue_copy(it + 1)
        e_end.record(stream)
        torch.cuda.synchronize()
        t_e2e = e_start.elapsed_time(e_end) * 1e-3
        if ws > 1:
            torch.distributed.barrier()
        e2e_rate, t_e2e = _job_rate(tokens_per_step * n_e2e, t_e2e, ws, dev)
        # The input copy alone (what the end-to-end rate overlaps with compute).
        c0 = torch.cuda.Event(enable_timing=True)
        c1 = torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(copy_stream):
            c0.record(copy_stream)
            for _ in range(5):
                dev_arenas[0].copy_(host_arena, non_blocking=True)
            c1.record(copy_stream)
        torch.cuda.synchronize()
        t_copy = c0.elapsed_time(c1) * 1e-3 / 5
        e2e = {"value": e2e_rate, "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "steps": n_e2e, "copies_per_step": {"h2d": 1, "d2h": 1},
               "h2d_copy_us": t_copy * 1e6, "h2d_gbs": h2d / t_copy / 1e9,
               "overlap": "inputs of step i+1 copied on a second stream while step i runs",
               "state_resident": "KV cache and W_lm stay in HBM (model state)"}

    # Kernel launches per step: attention, the accept call's one or two passes
    # (asked from the library), the separate commit if requested.
    n_acc_launches = spade.spade_accept_launches(B, R, wl["H"], wl["V"])

    # ---- the LM head's statistics pass alone (two-pass shapes) ----------------
    # It runs every LM-head flop; the sampling pass recomputes only the rows to
    # sample, and exits at once when no sequence samples.  So the accept call
    # with every sequence greedy times the statistics pass (plus that empty
    # second launch), after the timed region, L2 flushed between calls.
    pass1 = None
    if n_acc_launches == 2:
        greedy = torch.zeros_like(wl["mode"])
        acc_g = torch.zeros_like(acc)
        tok_g = torch.zeros_like(tok)
        ev1 = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(10)]
        _head_start(13)
        for i in range(13):
            if flush:
                flush_buf.zero_()
            if i >= 3:
                ev1[i - 3][0].record(stream)
            spade.spade_verify_accept(wl["hidden"], wl["w_lm"], wl["draft_tokens"], wl["draft_probs"],
                                      wl["uniforms"], greedy, wl["cu_q"], wl["n_draft"], acc_g, tok_g,
                                      workspace=ws_acc, status=status)
            if i >= 3:
                ev1[i - 3][1].record(stream)
        torch.cuda.synchronize()
        pass1 = statistics.median(a.elapsed_time(b) * 1e-3 for a, b in ev1)
    wl["ctx_lens"].copy_(ctx0)  # the step's commits advanced it
    qkv = _time_qkv(spec, wl, dev, flush_buf)
    hbm, bf16, bf16_sus, peak_src = _peaks()
    m_acc = statistics.mean(t_acc)
    m_attn = statistics.mean(t_attn)
    roof_lm = {"kernel": "verify_accept_kernel"}
    roof_lm.update(_lm_roofline(lm_bytes, lm_flop, m_acc, hbm, bf16_sus, bf16, peak_src))
    roof_lm["traffic"] = _traffic("verify_accept_kernel", args.workload)
    attn_kernel = "verify_attention_tc_kernel"
    roof_attn = {"kernel": attn_kernel, "bound": "hbm", "achieved": attn_bytes / m_attn / 1e9,
                 "peak": hbm, "unit": "GB/s", "frac": attn_bytes / m_attn / 1e9 / hbm,
                 "traffic": _traffic(attn_kernel, args.workload),
                 "algorithmic_bytes": attn_bytes, "peak_source": peak_src,
                 "tflops": attn_flop / m_attn / 1e12}
    dominant = roof_lm if m_acc >= m_attn else roof_attn
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": total / args.steps * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": _config(spec, wl_cpu, ws),
        "tokens_per_step": tokens_per_step,
        "accepted_len": acc.tolist(),
        "kernels_us": ({"verify_attention": m_attn * 1e6, "verify_accept": m_acc * 1e6,
                        "kv_commit": statistics.mean(t_com) * 1e6} if args.separate_commit else
                       {"verify_attention": m_attn * 1e6, "verify_accept_commit": m_acc * 1e6}),
        "roofline": dominant, "roofline_attention": roof_attn, "roofline_lm_head": roof_lm,
        "e2e": e2e, "gpu_launches": (1 + n_acc_launches + (1 if args.separate_commit else 0)) * args.steps,
        "wall_s_timed_loop": t_wall,
        "clocks": clk.summary(),
    }
    if qkv is not None:
        line["qkv_rope"] = qkv
    if pass1 is not None:
        line["lm_head_pass1"] = {"us": pass1 * 1e6, "tensor_tflops": lm_flop / pass1 / 1e12,
                                 "frac_of_sustained_bf16": lm_flop / pass1 / 1e12 / bf16_sus,
                                 "frac_of_burst_bf16": lm_flop / pass1 / 1e12 / bf16, "peak_source": peak_src,
                                 "how": "accept call with every sequence greedy (the sampling pass exits at once)"}
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        base, par = cpu_baseline(wl_cpu, acc.cpu(), tok.cpu())
        line["cpu_baseline"] = base
        line["parity"] = par
    if rank == 0 and ws == 1 and not args.no_sampling and spade.spade_accept_launches(
            wl["B"], wl["R"], wl["H"], wl["V"]) == 1:
        line["sampling"] = sampling_report(wl, dev)
    if rank == 0 and ws == 1 and not args.no_loop:
        line["speculative_loop"] = loop_report(dev)
    if rank == 0 and ws == 1 and not args.no_per_workload:
        line["per_workload"] = per_workload(args, dev, skip=args.workload)
    return line


# ---------------------------------------------------------------------------
def _time_qkv(spec, wl, dev, flush_buf=None, launches=20):
    """The verify block's QKV projection + rotary embedding (writes the K/V of the verify
    slots, as the step's attention expects them): median CUDA-event time per launch, L2
    flushed before each launch (W of a layer fits in L2), and its HBM roofline."""
    import paper_2608_13076_gb300 as spade

    x, w = W.make_qkv_inputs(spec, wl["R"], device=dev)
    q = torch.empty((wl["R"], wl["Hq"], wl["D"]), dtype=torch.bfloat16, device=dev)
    status = spade.status_tensor(dev)
    if flush_buf is None:
        flush_buf = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device=dev)
    kc, vc = wl["k_cache"].clone(), wl["v_cache"].clone()  # the step's caches stay as they were
    stream = torch.cuda.current_stream()
    max_k = int(wl["n_draft"].max())  # read once: a device read inside the loop would synchronise it
    ws = spade.qkv_workspace(wl["R"], wl["Hq"], wl["Hkv"], wl["D"], device=dev)

    def call():
        spade.spade_verify_qkv_rope(x, w, wl["ctx_lens"], wl["n_draft"], wl["cu_q"], q, kc, vc, Hq=wl["Hq"],
                                    Hkv=wl["Hkv"], rope_theta=spec.rope_theta, max_k=max_k, workspace=ws,
                                    status=status)

    # The first launch of a shape also runs one-time host work (occupancy queries):
    # finish it before the timed loop, which must not wait on the host.
    call()
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(launches)]
    _head_start(launches + 3)
    for i in range(launches + 3):
        flush_buf.zero_()
        if i >= 3:
            ev[i - 3][0].record(stream)
        call()
        if i >= 3:
            ev[i - 3][1].record(stream)
    torch.cuda.synchronize()
    if int(status.item()):
        raise RuntimeError(f"qkv_rope device status {int(status.item())}")
    t = statistics.median(a.elapsed_time(b) * 1e-3 for a, b in ev)
    hbm = _peaks()[0]
    R, H, Hq, Hkv, D = wl["R"], wl["H"], wl["Hq"], wl["Hkv"], wl["D"]
    nbytes = (Hq + 2 * Hkv) * D * H * 2 + R * H * 2 + R * (Hq + 2 * Hkv) * D * 2
    flop = 2.0 * R * (Hq + 2 * Hkv) * D * H
    return {"kernel": "qkv_rope_kernel", "us": t * 1e6, "bound": "hbm", "achieved": nbytes / t / 1e9, "peak": hbm,
            "unit": "GB/s", "frac": nbytes / t / 1e9 / hbm, "algorithmic_bytes": nbytes, "tflops": flop / t / 1e12,
            "traffic": _traffic("qkv_rope_kernel", spec.name),
            "launches": launches, "l2": "flushed before each launch",
            "note": "not part of the timed step (the step's q and cache slots are inputs); measured after it"}


def _time_step(wl, dev, steps, warmup):
    """Device time of the step (attention, then accept + commit) on one workload."""
    import paper_2608_13076_gb300 as spade

    B, R = wl["B"], wl["R"]
    max_k = int(wl["n_draft"].max())
    out = torch.empty_like(wl["q"])
    acc = torch.zeros(B, dtype=torch.int32, device=dev)
    tok = torch.zeros(B, dtype=torch.int32, device=dev)
    status = spade.status_tensor(dev)
    ws_attn = spade.attn_workspace(B, wl["Hq"], wl["Hkv"], wl["D"], wl["cap"], max_k, device=dev)
    ws_acc = spade.accept_workspace(B, R, wl["H"], wl["V"], device=dev)
    ctx0 = wl["ctx_lens"].clone()
    attn_bytes, lm_bytes, lm_flop, _, _ = _work_bytes(wl)
    flush = attn_bytes + lm_bytes < 2 * L2_BYTES
    flush_buf = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device=dev) if flush else None
    stream = torch.cuda.current_stream()
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    for s in range(warmup + steps):
        if s == 1:
            # The first step of a shape runs one-time host work; the timed steps must not
            # wait on the host, so the GPU gets a head start after it.
            torch.cuda.synchronize()
            _head_start(warmup + steps)
        wl["ctx_lens"].copy_(ctx0)
        if flush:
            flush_buf.zero_()
        e = evs[s - warmup] if s >= warmup else None
        if e:
            e[0].record(stream)
        spade.spade_verify_attention(wl["q"], wl["k_cache"], wl["v_cache"], wl["ctx_lens"], wl["n_draft"],
                                     wl["cu_q"], out, None, max_k=max_k, workspace=ws_attn, status=status)
        if e:
            e[1].record(stream)
        spade.spade_verify_accept_commit(wl["hidden"], wl["w_lm"], wl["draft_tokens"], wl["draft_probs"],
                                         wl["uniforms"], wl["mode"], wl["cu_q"], wl["n_draft"], acc, tok,
                                         wl["k_cache"], wl["v_cache"], wl["ctx_lens"], workspace=ws_acc,
                                         status=status)
        if e:
            e[2].record(stream)
    torch.cuda.synchronize()
    if int(status.item()) & ~spade.DEV_FALLBACK:
        raise RuntimeError(f"device status {int(status.item())} on {wl['spec'].name}")
    wl["ctx_lens"].copy_(ctx0)  # the commits advanced it
    t_attn = statistics.median(e[0].elapsed_time(e[1]) * 1e-3 for e in evs)
    t_acc = statistics.median(e[1].elapsed_time(e[2]) * 1e-3 for e in evs)
    return t_attn, t_acc, int((acc.long() + 1).sum().item()), acc.tolist()


def per_workload(args, dev, skip):
    """Device timing of every other workload of the suite (no end-to-end leg, no oracle)."""
    hbm, bf16, bf16_sus, peak_src = _peaks()
    res = {}
    for name, spec in W.SPECS.items():
        if name == skip:
            continue
        wl = _to_device(W.make_workload(spec, device="cpu"), dev)
        attn_bytes, lm_bytes, lm_flop, _, _ = _work_bytes(wl)
        t_attn, t_acc, toks, acc = _time_step(wl, dev, args.per_workload_steps, 3)
        qkv = _time_qkv(spec, wl, dev, launches=10)
        lm = _lm_roofline(lm_bytes, lm_flop, t_acc, hbm, bf16_sus, bf16, peak_src)
        res[name] = {"tokens_per_s": toks / (t_attn + t_acc), "us_per_step": (t_attn + t_acc) * 1e6,
                     "tokens_per_step": toks, "accepted_len": acc,
                     "verify_attention_us": t_attn * 1e6, "attention_hbm_frac": attn_bytes / t_attn / 1e9 / hbm,
                     "verify_accept_commit_us": t_acc * 1e6, "lm_head_bound": lm["bound"],
                     "lm_head_frac": lm["frac"], "lm_head_tensor_frac_of_sustained": lm["tensor"]["frac_of_sustained"],
                     "qkv_rope_us": qkv["us"], "qkv_rope_hbm_frac": qkv["frac"],
                     "steps": args.per_workload_steps, "timing": "median of CUDA-event times per launch"}
        del wl
        torch.cuda.empty_cache()
    return res


def sampling_report(wl, dev, launches=20):
    """Device time of the LM-head + accept launch with the verifier's sampling options (no
    commit): p whole, temperature 0.8, top-p 0.9, and both, on every sequence of the step."""
    import paper_2608_13076_gb300 as spade

    B, R = wl["B"], wl["R"]
    acc = torch.zeros(B, dtype=torch.int32, device=dev)
    tok = torch.zeros(B, dtype=torch.int32, device=dev)
    status = spade.status_tensor(dev)
    ws_acc = spade.accept_workspace(B, R, wl["H"], wl["V"], device=dev)
    temp = torch.full((B,), 0.8, dtype=torch.float32, device=dev)
    top_p = torch.full((B,), 0.9, dtype=torch.float32, device=dev)
    _, lm_bytes, _, _, _ = _work_bytes(wl)
    flush_buf = torch.empty(2 * L2_BYTES, dtype=torch.uint8, device=dev) if lm_bytes < 2 * L2_BYTES else None
    stream = torch.cuda.current_stream()
    res = {"workload": wl["spec"].name, "launches": launches,
           "timing": "median of CUDA-event times per launch", "top_p": 0.9, "temperature": 0.8}
    for name, t, p in (("plain", None, None), ("temperature", temp, None), ("top_p", None, top_p),
                       ("temperature_top_p", temp, top_p)):
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(launches)]
        for i in range(3 + launches):
            if i == 1:
                torch.cuda.synchronize()
                _head_start(3 + launches)
            if flush_buf is not None:
                flush_buf.zero_()
            e = evs[i - 3] if i >= 3 else None
            if e:
                e[0].record(stream)
            spade.spade_verify_accept_sampling(wl["hidden"], wl["w_lm"], wl["draft_tokens"], wl["draft_probs"],
                                               wl["uniforms"], wl["mode"], wl["cu_q"], wl["n_draft"], acc, tok,
                                               workspace=ws_acc, status=status, temperature=t, top_p=p)
            if e:
                e[1].record(stream)
        torch.cuda.synchronize()
        res[name + "_us"] = statistics.median(e[0].elapsed_time(e[1]) * 1e3 for e in evs)
    if int(status.item()) & ~spade.DEV_FALLBACK:
        raise RuntimeError(f"device status {int(status.item())} in the sampling report")
    return res


def loop_report(dev, B=8, max_new=64):
    """Algorithm 1 with the toy verifier (one layer through the library) for draft lengths
    0 (plain decoding), 1, 2, 4, 8: verifier calls per generated token and the acceptance
    rate, greedy and stochastic -- the synthetic analogue of the paper's cloud-call counts."""
    import numpy as np

    from paper_2608_13076_gb300 import speculative as S

    ver = S.ToyVerifier(S.ToyConfig(), B, cap=2048, seed=3, device=dev)
    g = np.random.default_rng(4)
    prompts = [list(g.integers(0, ver.cfg.V - 1, size=int(n))) for n in g.integers(8, 64, size=B)]
    out = {"model": "toy verifier: V 2048, H 512, GQA 8/2, D 64, one layer; drafter: its residual path",
           "sequences": B, "max_new": max_new}
    for name, mode in (("greedy", S.GREEDY), ("stochastic", S.STOCHASTIC)):
        rows = []
        for d in (0, 1, 2, 4, 8):
            t0 = time.perf_counter()
            res = S.speculative_decode(ver, prompts, d=d, max_new=max_new, mode=mode, seed=11)
            wall = time.perf_counter() - t0
            toks = sum(len(t) for t in res.tokens)
            rows.append({"d": d, "verifier_calls": sum(res.calls_per_seq), "tokens": toks,
                         "tokens_per_call": toks / max(1, sum(res.calls_per_seq)),
                         "acceptance": res.accepted / res.drafted if res.drafted else None,
                         "batch_calls": res.calls, "wall_s": wall})
        out[name] = rows
    return out


def _npf(t):
    return None if t is None else (t.float().numpy() if t.dtype == torch.bfloat16 else t.numpy())


def _oracle_one_sequence(wl_cpu, b):
    """Runs the oracle's verify step (attention + LM head + accept + commit) on sequence b.

    Returns (committed tokens, seconds, the oracle's accept result for b)."""
    import oracle.spade_oracle as O

    cu = wl_cpu["cu_q"]
    r0, r1 = int(cu[b]), int(cu[b + 1])
    k = r1 - r0 - 1
    q = _npf(wl_cpu["q"][r0:r1])
    kc = _npf(wl_cpu["k_cache"][b:b + 1])
    vc = _npf(wl_cpu["v_cache"][b:b + 1])
    ctx = _npf(wl_cpu["ctx_lens"][b:b + 1])
    kd = [k]
    cu1 = [0, k + 1]
    t0 = time.perf_counter()
    O.verify_attention(q, kc, vc, ctx, kd, cu1)
    logits = O.lm_logits(_npf(wl_cpu["hidden"][r0:r1]), _npf(wl_cpu["w_lm"]))
    d0 = r0 - b
    dp = _npf(wl_cpu["draft_probs"][d0:d0 + k]) if wl_cpu["draft_probs"] is not None else None
    res = O.verify_accept(logits, _npf(wl_cpu["draft_tokens"][d0:d0 + k]), dp,
                          _npf(wl_cpu["uniforms"][r0:r1]), _npf(wl_cpu["mode"][b:b + 1]), cu1, kd)
    O.kv_commit(kc, vc, ctx, res["accepted_len"], kd)
    dt = time.perf_counter() - t0
    return int(res["accepted_len"][0]) + 1, dt, res


def _cores():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


CPU_BUDGET_S = 25.0


def cpu_baseline(wl_cpu, acc_gpu, tok_gpu):
    """The oracle on the benched step, sequence by sequence, until all are done or about
    25 s of CPU time is spent; also the parity of the GPU step's decisions on them."""
    toks, secs, per = 0, 0.0, []
    B = wl_cpu["B"]
    for b in range(B):
        t, dt, res = _oracle_one_sequence(wl_cpu, b)
        toks += t
        secs += dt
        per.append((b, dt, res))
        if secs > CPU_BUDGET_S:
            break
    n = len(per)
    times = [dt for _, dt, _ in per]
    base = {"value": toks / secs, "unit": UNIT, "cores": _cores(), "kind": "oracle",
            "sample": (f"sequences 0..{n - 1} of {B} of the workload ({toks} committed tokens), one at a time: "
                       f"attention of its k+1 rows x all heads, float64 LM head over the full vocabulary, "
                       f"accept, commit; {secs:.2f} s in all, per sequence mean {statistics.mean(times):.2f} s "
                       f"(min {min(times):.2f}, max {max(times):.2f})")}
    a_g, t_g = acc_gpu.numpy(), tok_gpu.numpy()
    flagged = mism = mism_flagged = 0
    acc_oracle = []
    for b, _, res in per:
        fl = bool(res["flag_decision"][0] or res["flag_sample"][0])
        bad = a_g[b] != res["accepted_len"][0] or t_g[b] != res["next_token"][0]
        flagged += fl
        mism += bad and not fl
        mism_flagged += bad and fl
        acc_oracle.append(int(res["accepted_len"][0]))
    par = {"sequences_checked": n, "of": B, "flagged": int(flagged), "mismatch_unflagged": int(mism),
           "mismatch_flagged": int(mism_flagged), "accepted_len_oracle": acc_oracle,
           "rule": "accepted length and next token bit-exact except at positions whose float64 top-2 logit "
                   "gap, |u - p/q| or sampled-edge margin is below 1e-3, or whose draw lies within the spread fp32 logit errors give the cumulative mass (flagged, counted here)"}
    return base, par


def run_reference(args):
    spec = W.SPECS[args.workload]
    wl = W.make_workload(spec, device="cpu")
    B = wl["B"]
    for s in range(args.warmup):
        _oracle_one_sequence(wl, s % B)
    toks, secs = 0, 0.0
    acc = [None] * B
    for s in range(args.steps):
        t, dt, res = _oracle_one_sequence(wl, s % B)
        toks += t
        secs += dt
        acc[s % B] = int(res["accepted_len"][0])
    value = toks / secs
    sample = (f"each step: one sequence of the {args.workload} workload through the float64 oracle "
              f"(attention of its k+1 rows x {spec.Hq} heads, LM head over {spec.V} vocab, accept, commit), "
              f"sequences in turn")
    return {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": 1, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": secs / args.steps * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": _config(spec, wl, 1),
        "accepted_len": acc,
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": _cores(), "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def _json_default(o):
    """numpy scalars (from the oracle's results) as plain numbers."""
    if hasattr(o, "item"):
        return o.item()
    raise TypeError(f"{type(o).__name__} is not JSON serializable")


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="spade", choices=["spade", "reference"])
    ap.add_argument("--workload", default="llama3_8b", choices=sorted(W.SPECS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-per-workload", action="store_true",
                    help="skip the device timing of the suite's other workloads")
    ap.add_argument("--per-workload-steps", type=int, default=20)
    ap.add_argument("--no-loop", action="store_true", help="skip the decoding-loop report")
    ap.add_argument("--no-sampling", action="store_true",
                    help="skip the timing of the temperature / top-p accept launches")
    ap.add_argument("--separate-commit", action="store_true",
                    help="run the KV commit as its own launch instead of inside the LM-head kernel")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3) if args.impl == "spade" else args.warmup
    ws, rank, local = _dist()
    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args), default=_json_default), flush=True)
        return
    if ws > 1:
        torch.cuda.set_device(local)
        torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", local))
    line = run_spade(args, ws, rank, local)
    if rank == 0:
        print(json.dumps(line, default=_json_default), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
