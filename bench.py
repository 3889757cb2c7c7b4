#!/usr/bin/env python3
"""Throughput of the Whisper-Flash speculative decode step on GB300.

One step = one wf_step over the active batch: the drafter's pass, the
target's verify pass over [anchor, c_1..c_8], the history ingest and the
accept/rollback (all rows of the hot path).  Proposals are teacher-forced
from the target's own greedy continuation (computed first on the GPU, untimed)
with seeded accept lengths, so acceptance is realistic although the weights
are random.  Sequences that finish are compacted away; when a whole job has
finished it is rewound to its post-prefill state (the acoustic keys/values
and the prompt's cache rows are kept) and decoded again.

Prints one JSON line.  --impl reference times the CPU oracle instead (on the
host cores, rank 0 only).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2609_32869_gb300 import synthetic as syn  # noqa: E402

METRIC = "draft+verify tokens/s at B=1/16/96; step µs; HBM GB/s vs peak"

WORKLOADS = {
    "large_b1": dict(cfg="LARGE", batch=1, budget=(200, 200), accept="uniform",
                     text="Whisper-large-shaped decoder (d=1280, 20 heads, FFN 5120, 32 layers, "
                          "vocab 51866, 448 positions), 2-layer drafter copied from target layers "
                          "0 and 31, batch 1, 1500-frame encoder output, 4-token prompt, "
                          "200-token transcript, accept length uniform 0..8"),
    "large_b16": dict(cfg="LARGE", batch=16, budget=(20, 220), accept="geometric",
                      text="large shapes, batch 16, transcript lengths uniform 20..220, "
                           "accept length geometric (mean 4) per sequence"),
    "large_b96": dict(cfg="LARGE", batch=96, budget=(10, 220), accept="geometric",
                      text="large shapes, batch 96, transcript lengths uniform 10..220, "
                           "sequences finish asynchronously and the batch compacts"),
    "tiny_b1": dict(cfg="TINY", batch=1, budget=(200, 200), accept="uniform",
                    text="Whisper-tiny-shaped decoder (d=384, 6 heads, FFN 1536, 4 layers, "
                         "vocab 51865), batch 1, accept length uniform 0..8"),
    # Temperature sampling (App. A.4): the drafter draws its own proposals and
    # the target applies the rejection rule with seeded Philox streams; no
    # teacher forcing, so the accepted lengths are whatever the random weights
    # give (reported in the line).
    "large_b32_t07": dict(cfg="LARGE", batch=32, budget=(220, 220), temperature=0.7,
                          text="large shapes, batch 32, temperature 0.7 speculative sampling "
                               "(drafter's own proposals, rejection rule), 220-token budget"),
    "large_b32_t10": dict(cfg="LARGE", batch=32, budget=(220, 220), temperature=1.0,
                          text="large shapes, batch 32, temperature 1.0 speculative sampling "
                               "(drafter's own proposals, rejection rule), 220-token budget"),
    # Depth-reduced cases for profiler captures: every kernel keeps the large
    # per-layer shapes and launch configuration; only the number of target
    # blocks shrinks so a capture holds a few GB and few launches.
    "large_b1_4l": dict(cfg="LARGE", layers=4, batch=1, budget=(40, 40), accept="uniform",
                        text="large per-layer shapes cut to 4 target blocks (profiling case), "
                             "batch 1, 40-token transcript, accept length uniform 0..8"),
    "large_b96_2l": dict(cfg="LARGE", layers=2, batch=96, budget=(20, 40), accept="geometric",
                         text="large per-layer shapes cut to 2 target blocks (profiling case), "
                              "batch 96, transcript lengths uniform 20..40"),
}


# DRAM bytes (read + write) per projection launch, averaged over one step's
# launch mix, from ncu captures of the depth-reduced profiling cases with the
# same per-layer shapes (profiles/dram_per_kernel_large_b1_4l.md and
# profiles/dram_per_kernel_large_b96_2l.md); None where no capture covers the
# workload's shapes.
GEMM_DRAM_BYTES_PER_LAUNCH = {"large_b1": 7.826e6, "large_b96": 13.17e6}


def aggregate_ranks(times, counts, world, device):
    """Whole-job figures over `world` replica ranks: each time is the maximum
    over ranks (the slowest rank bounds the job), each count the sum (every
    rank decodes its own sequences).  With world == 1 the values come back
    unchanged; otherwise every rank must call this with the same lengths."""
    import torch
    t = torch.tensor([float(x) for x in times], dtype=torch.float64, device=device)
    c = torch.tensor([float(x) for x in counts], dtype=torch.float64, device=device)
    if world > 1:
        import torch.distributed as dist
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        dist.all_reduce(c, op=dist.ReduceOp.SUM)
    return [float(x) for x in t.cpu()], [float(x) for x in c.cpu()]


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            mp = json.load(f)
        return float(mp["hbm_gbs"]), float(mp["bf16_tflops"]), "measured"
    except Exception:
        return 6800.0, 1900.0, "fallback"


def _cfg(name, layers=None):
    cfg = getattr(syn, name)
    if layers:
        import dataclasses
        taps = tuple(min(t, layers - 1) for t in (0, 1, 2, 3, 3))
        cfg = dataclasses.replace(cfg, name=f"{cfg.name}_{layers}l", n_layers=layers, taps=taps,
                                  draft_init_from=(0, layers - 1))
    return cfg


# ----------------------------------------------------------------- schedule --
class Schedule:
    """Host-side replay of the teacher-forced job: which proposals each step
    gets, how many tokens it must emit, and when sequences finish."""

    def __init__(self, cfg, g, budgets, accept):
        self.cfg, self.g, self.budgets, self.accept = cfg, g, budgets, accept
        self.B = len(g)
        self.restart()

    def restart(self):
        self.t = np.ones(self.B, np.int64)                 # tokens emitted so far
        self.R = np.array(self.budgets, np.int64) - 1
        self.done = np.array([self.R[b] <= 0 or self.g[b][0] == self.cfg.eos_id
                              for b in range(self.B)])
        self.s = 0

    def step(self):
        """Proposals [B, K] for the next step and the tokens each slot emits."""
        K, V, eos = self.cfg.block_k, self.cfg.vocab, self.cfg.eos_id
        forced = np.zeros((self.B, K), np.int32)
        emitted = np.zeros(self.B, np.int64)
        for b in range(self.B):
            if self.done[b]:
                continue
            g, t = self.g[b], int(self.t[b])
            k = int(max(0, min(K, self.R[b] - 1)))
            a = int(min(self.accept[self.s % len(self.accept), b], k))
            for j in range(K):
                forced[b, j] = g[t + j] if t + j < len(g) else 0
            if a < k:
                forced[b, a] = (g[t + a] + 1) % V
            out = g[t:t + a + 1]
            if eos in out:
                out = out[:out.index(eos) + 1]
            n = len(out)
            emitted[b] = n
            self.t[b] += n
            self.R[b] -= n
            if self.R[b] <= 0 or out[-1] == eos:
                self.done[b] = True
        self.s += 1
        return forced, emitted


def _clock_sampler(uuid):
    fields = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    out = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
    cmd = ["nvidia-smi", f"--query-gpu={fields}", "--format=csv,noheader,nounits", "-lms", "100"]
    if uuid:
        cmd += ["-i", uuid]
    try:
        proc = subprocess.Popen(cmd, stdout=out, stderr=subprocess.DEVNULL)
    except OSError:
        return None, out.name
    return proc, out.name


def _clock_summary(path):
    sm, mx, reasons = [], [], set()
    try:
        rows = [r.split(",") for r in open(path).read().strip().splitlines()]
    except OSError:
        rows = []
    names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
    for r in rows:
        r = [x.strip() for x in r]
        if len(r) < 9:
            continue
        try:
            sm.append(float(r[1]))
            mx.append(float(r[2]))
        except ValueError:
            continue
        for nm, v in zip(names, r[5:9]):
            if v.lower().startswith("active"):
                reasons.add(nm)
    return {"sm_mhz": statistics.median(sm) if sm else None,
            "sm_max_mhz": max(mx) if mx else None,
            "reasons": sorted(reasons), "samples": len(sm)}


# --------------------------------------------------------------- our path --
def step_weight_kv_bytes(cfg, B, L):
    """Algorithmic bytes of one step: every weight matrix the step reads (target
    and drafter blocks without the acoustic K/V projections, the history
    projection and the drafter's key/value rows it re-reads, the tied head in
    both passes) plus every cached key/value row read (acoustic memory of 32+2
    blocks, the target cache up to L+8, the drafter history up to L+8)."""
    d, F, V, T, nl, nd = cfg.d_model, cfg.d_ff, cfg.vocab, cfg.enc_frames, cfg.n_layers, cfg.n_draft_layers
    per_block = 6 * d * d + 2 * d * F
    weights = 2 * (nl * per_block + nd * per_block + cfg.n_taps * d * d + nd * 2 * d * d + 2 * V * d)
    cross = B * (nl + nd) * 2 * T * d * 2
    self_kv = sum((nl + nd) * 2 * (int(l) + cfg.block_k + 1) * d * 2 for l in L)
    return weights, cross + self_kv


def run_ours(args, rank, world):
    import torch
    import torch.distributed as dist
    from paper_2609_32869_gb300 import binding as B
    from paper_2609_32869_gb300.session import Session, upload_weights

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    wl = WORKLOADS[args.workload]
    cfg = _cfg(wl["cfg"], wl.get("layers"))
    Bn = wl["batch"]
    host_ws = syn.make_weights(cfg, seed=0)
    dev = upload_weights(host_ws)
    need_cpu = rank == 0 and world == 1 and not args.no_cpu_baseline
    if not need_cpu:
        host_ws = None
    enc = syn.encoder_output(cfg, Bn, seed=1)
    prompt = syn.prompts(cfg, Bn, length=4, seed=1)
    lo, hi = wl["budget"]
    if args.budget:
        lo = hi = args.budget
    budgets = np.full(Bn, lo, np.int32) if lo == hi else syn.budgets(Bn, lo, hi, seed=2)
    sess = Session(cfg, dev, max_batch=Bn, max_ctx=cfg.max_pos)
    if args.persist:
        B.wf_set_option(sess.h, B.WF_OPT_PERSIST, 1)
    slots = np.arange(Bn, dtype=np.int32)
    stream = sess.stream

    # prefill and the target's greedy continuation (untimed)
    first = sess.prefill(slots, enc, prompt, budgets).cpu().numpy()
    g = [[int(first[b])] for b in range(Bn)]
    while True:
        toks, cnt = sess.greedy_step()
        toks, cnt = toks.cpu().numpy(), cnt.cpu().numpy()
        if cnt.sum() == 0:
            break
        for b in range(Bn):
            g[b].extend(int(x) for x in toks[b, :cnt[b]])
    n_steps = args.warmup + args.steps
    if wl["accept"] == "uniform":
        acc = syn.accept_uniform(max(n_steps, 64), Bn, k=cfg.block_k, seed=3)
    else:
        acc = syn.accept_geometric(max(n_steps, 64), Bn, mean=4.0, k=cfg.block_k, seed=3)
    sched = Schedule(cfg, g, budgets, acc)

    d_slots = torch.as_tensor(slots, device="cuda")

    def restart_job():
        """Rewind every slot to its post-prefill state and re-activate it."""
        B.wf_reset_slots(sess.h, Bn, d_slots, stream)
        B.wf_compact(sess.h, stream)
        return 2

    def make_plan(n):
        """Host replay of n steps of the job from its start: proposals, whether
        the job restarts before a step, whether the batch compacts after it,
        and the tokens it emits."""
        sched.restart()
        forced = np.zeros((n, Bn, cfg.block_k), np.int32)
        pre, comp, toks, kv = [], [], [], []
        for i in range(n):
            restart = bool(sched.done.all())
            if restart:
                sched.restart()
            live = [4 + int(sched.t[b]) - 1 for b in range(Bn) if not sched.done[b]]
            kv.append(step_weight_kv_bytes(cfg, len(live), live)[1])
            f, em = sched.step()
            forced[i] = f
            pre.append(restart)
            comp.append(bool((em > 0).any() and sched.done[em > 0].any()))
            toks.append(int(em.sum()))
        lens = [4 + int(sched.t[b]) - 1 for b in range(Bn)]
        dev_forced = torch.as_tensor(forced).cuda()
        return dict(forced=forced, dev=dev_forced, pre=pre, comp=comp, toks=toks, lens=lens, kv=kv)

    def execute(pl, lo, hi, e2e=False, pin=None):
        launches = 0
        for i in range(lo, hi):
            if pl["pre"][i]:
                launches += restart_job()
            if e2e:
                pin["in"].copy_(torch.as_tensor(pl["forced"][i]))
                pin["dev_in"].copy_(pin["in"], non_blocking=True)
                B.wf_step(sess.h, None, pin["dev_in"], sess.out_tokens, sess.out_count, stream)
                launches += B.wf_last_launch_count(sess.h)
                pin["out_tok"].copy_(sess.out_tokens, non_blocking=True)
                pin["out_cnt"].copy_(sess.out_count, non_blocking=True)
                stream.synchronize()
            else:
                B.wf_step(sess.h, None, pl["dev"][i], sess.out_tokens, sess.out_count, stream)
                launches += B.wf_last_launch_count(sess.h)
            if pl["comp"][i]:
                B.wf_compact(sess.h, stream)
                launches += 1
        return launches

    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(local).uuid)
        if uuid and not uuid.startswith("GPU-"):
            uuid = "GPU-" + uuid
    except Exception:
        uuid = None
    sampler, clock_path = _clock_sampler(uuid)

    # ---- warm-up and the device-timed region (inputs already in HBM)
    pl = make_plan(n_steps)
    restart_job()
    execute(pl, 0, args.warmup)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if args.profile_region:
        torch.cuda.profiler.start()
    e0.record(stream)
    launches = execute(pl, args.warmup, n_steps)
    e1.record(stream)
    torch.cuda.synchronize()
    if args.profile_region:
        torch.cuda.profiler.stop()
    if world > 1:
        dist.barrier()
    dev_ms = e0.elapsed_time(e1)
    tokens = sum(pl["toks"][args.warmup:])
    state = sess.state()
    err = sess.error()
    consistent = bool(all(int(state["len"][b]) == pl["lens"][b] for b in range(Bn)) and err == 0)

    # ---- end to end through the C ABI: pinned host proposals in, tokens out
    Kc = cfg.block_k
    pin = {"in": torch.empty((Bn, Kc), dtype=torch.int32).pin_memory(),
           "dev_in": torch.empty((Bn, Kc), dtype=torch.int32, device="cuda"),
           "out_tok": torch.empty((Bn, Kc + 1), dtype=torch.int32).pin_memory(),
           "out_cnt": torch.empty((Bn,), dtype=torch.int32).pin_memory()}
    # the same steps as the device-timed region, after the same warm-up
    pl2 = make_plan(n_steps)
    restart_job()
    execute(pl2, 0, args.warmup)
    torch.cuda.synchronize()
    w0 = time.perf_counter()
    execute(pl2, args.warmup, n_steps, e2e=True, pin=pin)
    torch.cuda.synchronize()
    e2e_s = time.perf_counter() - w0
    e2e_tokens = sum(pl2["toks"][args.warmup:])

    # ---- per-family kernel time with CUDA events (roofline of the top kernel)
    n_prof = min(args.steps, 5)
    pl3 = make_plan(n_prof)
    restart_job()
    B.wf_set_option(sess.h, B.WF_OPT_PROFILE, 1)
    execute(pl3, 0, n_prof)
    prof = B.wf_profile_read(sess.h, stream)
    B.wf_set_option(sess.h, B.WF_OPT_PROFILE, 0)

    if sampler is not None:
        sampler.terminate()
        sampler.wait()
    clocks = _clock_summary(clock_path)
    try:
        os.unlink(clock_path)
    except OSError:
        pass

    # ---- aggregate over ranks
    (dev_ms, e2e_s), (tokens, e2e_tokens) = aggregate_ranks([dev_ms, e2e_s], [tokens, e2e_tokens], world, "cuda")

    hbm_peak, bf16_peak, peak_src = _peaks()
    step_ms = dev_ms / args.steps
    wbytes = step_weight_kv_bytes(cfg, 0, [])[0]
    kvbytes = float(np.mean(pl["kv"][args.warmup:]))
    fam = max(("gemm", "head", "attn_cross", "attn_self", "persist"), key=lambda f: prof[f]["ms"])
    roof_fam = "persist" if args.persist else "gemm"
    fam_ms = prof[roof_fam]["ms"]
    gemm_gbs = prof[roof_fam]["bytes"] / (fam_ms * 1e-3) / 1e9 if fam_ms > 0 else None
    step_total_prof = sum(v["ms"] for v in prof.values())
    result = {
        "metric": METRIC,
        "value": tokens / (dev_ms * 1e-3),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": step_ms,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded random weights and encoder outputs; proposals teacher-forced "
                "from the target's own greedy continuation)",
        "config": {"workload": args.workload, "description": wl["text"], "batch": Bn,
                   "block": cfg.block_k + 1, "parallelism": f"replicas x{world}",
                   "path": "persistent passes" if args.persist else "launch by launch",
                   "l2": "inputs larger than L2 (every step streams "
                         f"{(wbytes + kvbytes) / 1e9:.2f} GB of weights and K/V > 129 MB L2)"},
        "step_us": step_ms * 1e3,
        "tokens_per_step": tokens / args.steps / world,
        "step_roofline": {"bytes": wbytes + kvbytes, "weights": wbytes, "kv": kvbytes,
                          "achieved_gbs": (wbytes + kvbytes) / (step_ms * 1e-3) / 1e9,
                          "peak_gbs": hbm_peak,
                          "frac": (wbytes + kvbytes) / (step_ms * 1e-3) / 1e9 / hbm_peak,
                          "peak_source": f"{peak_src} (MEASURED_PEAKS hbm_gbs)"},
        "roofline": {"kernel": ("persist_kernel (every block of a pass in one launch; bytes = weights "
                                "and acoustic K/V)") if args.persist else "gemm_tc_kernel (tcgen05 projections)",
                     "bound": "hbm",
                     "achieved": gemm_gbs, "peak": hbm_peak, "unit": "GB/s",
                     "frac": gemm_gbs / hbm_peak if gemm_gbs else None,
                     "traffic": None if args.persist else GEMM_DRAM_BYTES_PER_LAUNCH.get(args.workload),
                     "peak_source": peak_src,
                     "measured": f"CUDA events around each launch over {n_prof} profiled steps",
                     "share_of_kernel_time": fam_ms / step_total_prof if step_total_prof else None},
        "kernel_families_ms_per_step": {k: v["ms"] / n_prof for k, v in prof.items()},
        "kernel_families_launches_per_step": {k: v["launches"] / n_prof for k, v in prof.items()},
        "top_family": fam,
        "e2e": {"value": e2e_tokens / e2e_s, "unit": "tokens/s",
                "h2d_bytes_per_step": Bn * Kc * 4,
                "d2h_bytes_per_step": Bn * (Kc + 1) * 4 + Bn * 4},
        "gpu_launches": launches,
        "clocks": clocks,
        "consistent": consistent,
        "device_error": err,
    }
    if need_cpu:
        result["cpu_baseline"] = cpu_baseline(cfg, host_ws, enc, prompt, budgets, acc,
                                              budget_s=args.cpu_seconds)
    return result


def run_sampling(args, rank, world):
    """Speculative sampling steps: tokens/s from the counts the step itself
    returns (written per step into a device array, read after the region)."""
    import torch
    import torch.distributed as dist
    from paper_2609_32869_gb300 import binding as B
    from paper_2609_32869_gb300.session import Session, upload_weights

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    wl = WORKLOADS[args.workload]
    cfg = _cfg(wl["cfg"], wl.get("layers"))
    Bn, Kc = wl["batch"], cfg.block_k
    dev = upload_weights(syn.make_weights(cfg, seed=0))
    enc = syn.encoder_output(cfg, Bn, seed=1)
    prompt = syn.prompts(cfg, Bn, length=4, seed=1)
    budgets = np.full(Bn, wl["budget"][0], np.int32)
    sess = Session(cfg, dev, max_batch=Bn, max_ctx=cfg.max_pos)
    stream = sess.stream
    sp = B.sample_params(wl["temperature"], 4 + rank)
    sess.prefill(np.arange(Bn, dtype=np.int32), enc, prompt, budgets, sp=sp)
    n_steps = args.warmup + args.steps
    counts = torch.zeros(n_steps, Bn, dtype=torch.int32, device="cuda")
    toks = torch.zeros(n_steps, Bn, Kc + 1, dtype=torch.int32, device="cuda")

    def run(lo, hi):
        n = 0
        for i in range(lo, hi):
            B.wf_step(sess.h, sp, None, toks[i], counts[i], stream)
            n += B.wf_last_launch_count(sess.h)
        return n

    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(local).uuid)
        if uuid and not uuid.startswith("GPU-"):
            uuid = "GPU-" + uuid
    except Exception:
        uuid = None
    sampler, clock_path = _clock_sampler(uuid)
    run(0, args.warmup)
    torch.cuda.synchronize()
    len0 = sess.state()["len"].astype(np.float64)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if args.profile_region:
        torch.cuda.profiler.start()
    e0.record(stream)
    launches = run(args.warmup, n_steps)
    e1.record(stream)
    torch.cuda.synchronize()
    if args.profile_region:
        torch.cuda.profiler.stop()
    if world > 1:
        dist.barrier()
    dev_ms = e0.elapsed_time(e1)
    len1 = sess.state()["len"].astype(np.float64)
    c = counts[args.warmup:].cpu().numpy()
    tokens = float(c.sum())
    live = c > 0
    accepted = float((c[live] - 1).mean()) if live.any() else 0.0

    # end to end: the same call with the step's outputs read back to pinned
    # host memory every step (the step takes no per-step input)
    h_tok = torch.empty((Bn, Kc + 1), dtype=torch.int32).pin_memory()
    h_cnt = torch.empty((Bn,), dtype=torch.int32).pin_memory()
    e2e_tokens = 0
    torch.cuda.synchronize()
    w0 = time.perf_counter()
    for i in range(args.warmup, n_steps):
        B.wf_step(sess.h, sp, None, toks[i], counts[i], stream)
        h_tok.copy_(toks[i], non_blocking=True)
        h_cnt.copy_(counts[i], non_blocking=True)
        stream.synchronize()
        e2e_tokens += int(h_cnt.sum())
    e2e_s = time.perf_counter() - w0

    n_prof = min(args.steps, 3)
    B.wf_set_option(sess.h, B.WF_OPT_PROFILE, 1)
    run(0, n_prof)
    prof = B.wf_profile_read(sess.h, stream)
    B.wf_set_option(sess.h, B.WF_OPT_PROFILE, 0)
    if sampler is not None:
        sampler.terminate()
        sampler.wait()
    clocks = _clock_summary(clock_path)
    try:
        os.unlink(clock_path)
    except OSError:
        pass

    (dev_ms, e2e_s), (tokens, e2e_tokens) = aggregate_ranks([dev_ms, e2e_s], [tokens, e2e_tokens], world, "cuda")
    hbm_peak, _, peak_src = _peaks()
    step_ms = dev_ms / args.steps
    mean_len = list((len0 + len1) / 2.0)
    wbytes, kvbytes = step_weight_kv_bytes(cfg, Bn, [int(x) for x in mean_len])
    fam_ms = prof["gemm"]["ms"]
    gemm_gbs = prof["gemm"]["bytes"] / (fam_ms * 1e-3) / 1e9 if fam_ms > 0 else None
    return {
        "metric": METRIC,
        "value": tokens / (dev_ms * 1e-3),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": step_ms,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded random weights and encoder outputs; the drafter's own "
                "sampled proposals)",
        "config": {"workload": args.workload, "description": wl["text"], "batch": Bn,
                   "block": Kc + 1, "temperature": wl["temperature"],
                   "parallelism": f"replicas x{world}",
                   "l2": "inputs larger than L2 (every step streams "
                         f"{(wbytes + kvbytes) / 1e9:.2f} GB of weights and K/V > 129 MB L2)"},
        "step_us": step_ms * 1e3,
        "tokens_per_step": tokens / args.steps / world,
        "accepted_drafts_per_sequence_step": accepted,
        "step_roofline": {"bytes": wbytes + kvbytes, "weights": wbytes, "kv": kvbytes,
                          "achieved_gbs": (wbytes + kvbytes) / (step_ms * 1e-3) / 1e9,
                          "peak_gbs": hbm_peak,
                          "frac": (wbytes + kvbytes) / (step_ms * 1e-3) / 1e9 / hbm_peak,
                          "peak_source": f"{peak_src} (MEASURED_PEAKS hbm_gbs)"},
        "roofline": {"kernel": "gemm_tc_kernel (tcgen05 projections)", "bound": "hbm",
                     "achieved": gemm_gbs, "peak": hbm_peak, "unit": "GB/s",
                     "frac": gemm_gbs / hbm_peak if gemm_gbs else None,
                     "traffic": GEMM_DRAM_BYTES_PER_LAUNCH.get(args.workload),
                     "peak_source": peak_src,
                     "measured": f"CUDA events around each launch over {n_prof} profiled steps"},
        "kernel_families_ms_per_step": {k: v["ms"] / n_prof for k, v in prof.items()},
        "e2e": {"value": e2e_tokens / e2e_s, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": Bn * (Kc + 1) * 4 + Bn * 4},
        "gpu_launches": launches,
        "clocks": clocks,
        "device_error": sess.error(),
    }


# ------------------------------------------------------------ CPU oracle ----
def _oracle_setup(cfg, ws, enc, prompt, budgets):
    from oracle.decoder import WhisperFlashOracle
    o = WhisperFlashOracle(syn.weights_as_float(ws, np.float64), cfg)
    encf = syn.bf16_bits_to_f32(enc[0]).astype(np.float64)
    return o, encf


def _rewind(seq, L, anchor, remaining, emitted_len, step):
    """Drop cache rows past L (the oracle keeps accepted rows only)."""
    seq.self_k = [k[:L] for k in seq.self_k]
    seq.self_v = [v[:L] for v in seq.self_v]
    seq.hist = seq.hist[:L]
    seq.L, seq.anchor, seq.remaining = L, anchor, remaining
    seq.emitted = seq.emitted[:emitted_len]
    seq.done = False
    seq.step = step


def _oracle_run(cfg, ws, enc, prompt, budgets, acc, n_warm, n_steps, prefix_tokens=40,
                time_cap_s=None):
    """The oracle decodes sequence 0 of the workload: prefill (untimed), the
    first `prefix_tokens` tokens of its own greedy continuation (untimed; they
    supply the teacher-forced proposals), then speculative steps with the
    schedule's accept lengths, rewinding to the post-prefill state whenever
    that prefix is used up.  Returns (tokens, seconds, timed steps)."""
    o, encf = _oracle_setup(cfg, ws, enc, prompt, budgets)
    budget = int(budgets[0])
    seq = o.prefill(encf, prompt[0], budget, seq_id=0)
    L0, a0, R0, s0 = seq.L, seq.anchor, seq.remaining, seq.step
    need = min(prefix_tokens, budget)
    while len(seq.emitted) < need and not seq.done:
        o.greedy_step(seq)
    g = list(seq.emitted)
    _rewind(seq, L0, a0, R0, 1, s0)
    sched = Schedule(cfg, [g], [len(g)], acc)
    tokens, secs, done_steps = 0, 0.0, 0
    for i in range(n_warm + n_steps):
        if sched.done.all():
            _rewind(seq, L0, a0, len(g) - 1, 1, s0)
            sched.restart()
        forced, em = sched.step()
        seq.remaining = int(sched.R[0] + em[0])      # the prefix is the transcript here
        t0 = time.perf_counter()
        rec = o.spec_step(seq, forced=forced[0])
        dt = time.perf_counter() - t0
        if i >= n_warm:
            tokens += len(rec.emitted)
            secs += dt
            done_steps += 1
            if time_cap_s is not None and secs >= time_cap_s:
                break
    return tokens, secs, done_steps


def _cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def cpu_baseline(cfg, ws, enc, prompt, budgets, acc, budget_s=15.0):
    tokens, secs, steps = _oracle_run(cfg, ws, enc, prompt, budgets, acc, 0, 64,
                                      prefix_tokens=24, time_cap_s=budget_s)
    return {"value": tokens / secs, "unit": "tokens/s", "cores": _cores(), "kind": "oracle",
            "sample": f"{steps} teacher-forced speculative steps of sequence 0 over the first "
                      f"24 tokens of its transcript (float64 numpy oracle; prefill and the "
                      f"oracle's own greedy prefix untimed), {tokens} tokens in {secs:.1f} s",
            "ms_per_step": secs / steps * 1e3}


def _oracle_sampling_run(cfg, ws, enc, prompt, budget, T, n_warm, n_steps, time_cap_s):
    """The oracle's own speculative sampling of sequence 0 (drafter proposals,
    rejection rule) with the same Philox streams as the GPU run."""
    o, encf = _oracle_setup(cfg, ws, enc, prompt, [budget])
    seq = o.prefill(encf, prompt[0], budget, seq_id=0, temperature=T, seed=4)
    tokens, secs, done_steps = 0, 0.0, 0
    for i in range(n_warm + n_steps):
        if seq.done:
            break
        t0 = time.perf_counter()
        rec = o.spec_step(seq, temperature=T, seed=4)
        dt = time.perf_counter() - t0
        if i >= n_warm:
            tokens += len(rec.emitted)
            secs += dt
            done_steps += 1
            if secs >= time_cap_s:
                break
    return tokens, secs, done_steps


def run_reference(args):
    wl = WORKLOADS[args.workload]
    cfg = _cfg(wl["cfg"], wl.get("layers"))
    ws = syn.make_weights(cfg, seed=0)
    Bn = wl["batch"]
    enc = syn.encoder_output(cfg, 1, seed=1)
    prompt = syn.prompts(cfg, 1, length=4, seed=1)
    lo, hi = wl["budget"]
    budgets = np.full(Bn, lo, np.int32) if lo == hi else syn.budgets(Bn, lo, hi, seed=2)
    if wl.get("temperature"):
        tokens, secs, steps = _oracle_sampling_run(cfg, ws, enc, prompt, int(budgets[0]),
                                                   wl["temperature"], min(args.warmup, 3),
                                                   args.steps, args.cpu_seconds * 4)
        v = tokens / secs
        return {"impl": "reference", "metric": METRIC, "value": v, "unit": "tokens/s",
                "n_gpus": 1, "steps": steps, "warmup": args.warmup,
                "ms_per_step": secs / steps * 1e3, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                "config": {"workload": args.workload, "description": wl["text"], "batch": 1,
                           "block": cfg.block_k + 1, "temperature": wl["temperature"]},
                "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": _cores(),
                                 "kind": "oracle",
                                 "sample": f"{steps} speculative sampling steps of one sequence "
                                           f"(float64 numpy oracle; prefill untimed)"},
                "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}}
    if wl["accept"] == "uniform":
        acc = syn.accept_uniform(max(args.warmup + args.steps, 64), Bn, k=cfg.block_k, seed=3)
    else:
        acc = syn.accept_geometric(max(args.warmup + args.steps, 64), Bn, mean=4.0,
                                   k=cfg.block_k, seed=3)
    tokens, secs, steps = _oracle_run(cfg, ws, enc, prompt, budgets, acc, min(args.warmup, 3),
                                      args.steps, prefix_tokens=40, time_cap_s=args.cpu_seconds * 4)
    v = tokens / secs
    return {"impl": "reference", "metric": METRIC, "value": v, "unit": "tokens/s",
            "n_gpus": 1, "steps": steps, "warmup": args.warmup, "ms_per_step": secs / steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": args.workload, "description": wl["text"],
                                            "batch": 1, "block": cfg.block_k + 1},
            "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": _cores(), "kind": "oracle",
                             "sample": f"{steps} teacher-forced speculative steps of one "
                                       f"sequence over the first 40 tokens of its transcript "
                                       f"(float64 numpy oracle; greedy prefix untimed)"},
            "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--workload", choices=tuple(WORKLOADS), default="large_b1")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--profile-region", action="store_true",
                    help="cudaProfilerStart/Stop around the timed steps (for ncu)")
    ap.add_argument("--budget", type=int, default=0,
                    help="override every transcript budget (short profiling runs)")
    ap.add_argument("--persist", action="store_true",
                    help="run every drafter, verify and greedy pass as one persistent launch "
                         "(WF_OPT_PERSIST; batch * 9 <= 16 only)")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "reference":
        if rank != 0:
            return 0
        print(json.dumps(run_reference(args)), flush=True)
        return 0
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    if WORKLOADS[args.workload].get("temperature"):
        res = run_sampling(args, rank, world)
    else:
        res = run_ours(args, rank, world)
    if rank == 0:
        print(json.dumps(res), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
