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
    # Temperature sampling (App. A.4): proposals drawn from a seeded softmax over
    # perturbed target logits along the target's own sampled path, passed with
    # the logits of that distribution; the target applies the rejection rule
    # with seeded Philox streams.
    "large_b32_t07": dict(cfg="LARGE", batch=32, budget=(20, 220), temperature=0.7, sigma=0.3,
                          text="large shapes, batch 32, temperature 0.7 speculative sampling; "
                               "proposals from softmax((z_target + 0.3 eps) / T), eps ~ N(0, 1) seeded, "
                               "along the target's own sampled path; lengths uniform 20..220"),
    "large_b32_t10": dict(cfg="LARGE", batch=32, budget=(20, 220), temperature=1.0, sigma=0.3,
                          text="large shapes, batch 32, temperature 1.0 speculative sampling; "
                               "proposals from softmax((z_target + 0.3 eps) / T), eps ~ N(0, 1) seeded, "
                               "along the target's own sampled path; lengths uniform 20..220"),
    # Depth-reduced cases for profiler captures: every kernel keeps the large
    # per-layer shapes and launch configuration; only the number of target
    # blocks shrinks so a capture holds a few GB and few launches.
    "large_b1_4l": dict(cfg="LARGE", layers=4, batch=1, budget=(40, 40), accept="uniform",
                        text="large per-layer shapes cut to 4 target blocks (profiling case), "
                             "batch 1, 40-token transcript, accept length uniform 0..8"),
    "large_b96_2l": dict(cfg="LARGE", layers=2, batch=96, budget=(20, 40), accept="geometric",
                         text="large per-layer shapes cut to 2 target blocks (profiling case), "
                              "batch 96, transcript lengths uniform 20..40"),
    "large_b16_2l": dict(cfg="LARGE", layers=2, batch=16, budget=(20, 40), accept="geometric",
                         text="large per-layer shapes cut to 2 target blocks (profiling case), "
                              "batch 16, transcript lengths uniform 20..40"),
}


# DRAM bytes (read + write) per projection launch, averaged over one step's
# launch mix, from ncu captures of the depth-reduced profiling cases with the
# same per-layer shapes (profiles/dram_per_kernel_large_b1_4l.md,
# profiles/dram_per_kernel_large_b16_2l.md and
# profiles/dram_per_kernel_large_b96_2l.md); None where no capture covers the
# workload's shapes and projection path.
GEMM_DRAM_BYTES_PER_LAUNCH = {
    # 68 x out/cross-out (3.404 MB), 34 x fc1 (13.219), 34 x fc2 (13.313),
    # 2 x history K/V (6.662), 1 x history projection (16.572) per step
    "large_b1": 8.370e6,
    # 34 x QKV (12.077 MB), 102 x out/cross-out/fc2 (15.296), 34 x cross-query
    # (5.514), 34 x fc1 (15.354), 2 x history K/V (8.796), 1 x history
    # projection (27.283) per step, captured at 94 sequences
    "large_b96": 13.165e6,
    # 204 x batched skinny projections (8.593 MB), 2 x history K/V (7.346), 1 x
    # history projection (18.194) per step, captured at 15 live sequences with
    # --skinny (the default batch-16 path is tcgen05, which no capture covers)
    "large_b16": 8.627e6,
}

# the projection path each capture above ran on (its traffic describes only that path)
GEMM_DRAM_CAPTURE_PATH = {"large_b1": "skinny", "large_b16": "skinny", "large_b96": "tcgen05"}


def _gemm_traffic(name, path):
    return GEMM_DRAM_BYTES_PER_LAUNCH.get(name) if GEMM_DRAM_CAPTURE_PATH.get(name) == path else None


def _proj_kernel(path, rows):
    """The kernel that runs a pass's projections: the skinny kernels up to 144
    step rows (one operand tile up to 14), else the tcgen05 GEMM."""
    if path != "skinny":
        return "gemm_tc_kernel (tcgen05 projections)"
    if rows <= 14:
        return "skinny_kernel (single-sequence projections)"
    return "skinny_mt_kernel (batched skinny projections)"


# Tensor-pipe activity of the projections at batch 96 from the committed ncu
# capture of the same kernels (profiles/), or absent until one is taken.
TENSOR_PIPE_FROM_PROFILE = {
    "large_b96": {"pct_of_peak_elapsed_time_weighted": 7.8,
                  "by_projection": {"fc1": 12.0, "QKV": 9.1, "cross_query": 6.2,
                                    "out_crossout_fc2": 5.7, "history_kv": 10.1},
                  "source": "profiles/dram_per_kernel_large_b96_2l.md (ncu, 94 sequences, 2 target blocks)"},
}


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


def _device_uuid(local):
    import torch
    try:
        uuid = str(torch.cuda.get_device_properties(local).uuid)
        return uuid if uuid.startswith("GPU-") else "GPU-" + uuid
    except Exception:
        return None


def _family_roofline(prof, n_prof, step_ms, fam, hbm_peak, peak_src, kernel, traffic):
    """Roofline of one kernel family.  The family's share of the step comes from
    CUDA events around each launch (which serialise the launches), and its time
    per step is that share of the device-timed step, so it never exceeds the
    step; achieved = the family's algorithmic bytes per step / that time."""
    total = sum(v["ms"] for v in prof.values())
    share = prof[fam]["ms"] / total if total > 0 else None
    launches = prof[fam]["launches"] / n_prof
    if not share or not launches:
        return None
    fam_ms = share * step_ms
    bytes_step = prof[fam]["bytes"] / n_prof
    achieved = bytes_step / (fam_ms * 1e-3) / 1e9
    return {"kernel": kernel, "bound": "hbm", "achieved": achieved, "peak": hbm_peak, "unit": "GB/s",
            "frac": achieved / hbm_peak, "traffic": traffic, "peak_source": peak_src,
            "algorithmic_bytes_per_launch": bytes_step / launches,
            "launches_per_step": launches, "share_of_step": share,
            "us_per_launch": fam_ms * 1e3 / launches,
            "measured": f"share of CUDA-event kernel time over {n_prof} profiled steps x the "
                        f"device-timed ms_per_step"}


def measure_greedy(args, wl_name, dev, host_ws, rank, world, steps, warmup, e2e=True):
    """Teacher-forced speculative steps of one workload: device-timed region,
    optionally the same steps end to end, and per-family kernel time."""
    import torch
    import torch.distributed as dist
    from paper_2609_32869_gb300 import binding as B
    from paper_2609_32869_gb300.session import Session

    wl = WORKLOADS[wl_name]
    cfg = _cfg(wl["cfg"], wl.get("layers"))
    Bn = wl["batch"]
    enc = syn.encoder_output(cfg, Bn, seed=1)
    prompt = syn.prompts(cfg, Bn, length=4, seed=1)
    lo, hi = wl["budget"]
    if args.budget:
        lo = hi = args.budget
    budgets = np.full(Bn, lo, np.int32) if lo == hi else syn.budgets(Bn, lo, hi, seed=2)
    sess = Session(cfg, dev, max_batch=Bn, max_ctx=cfg.max_pos)
    if args.persist:
        B.wf_set_option(sess.h, B.WF_OPT_PERSIST, 1)
    # the library's default form: skinny projections for single-sequence
    # handles, tcgen05 above (--skinny: the batched skinny form up to 144 rows)
    proj_path = "tcgen05"
    if args.no_skinny:
        B.wf_set_option(sess.h, B.WF_OPT_SKINNY, 0)
    elif Bn * (cfg.block_k + 1) <= 14 or args.skinny:
        try:
            B.wf_set_option(sess.h, B.WF_OPT_SKINNY, 1)
            proj_path = "skinny"
        except B.WfError:
            pass
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
    n_steps = warmup + steps
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
        pre, comp, toks, kv, ctx = [], [], [], [], []
        for i in range(n):
            restart = bool(sched.done.all())
            if restart:
                sched.restart()
            live = [4 + int(sched.t[b]) - 1 for b in range(Bn) if not sched.done[b]]
            kv.append(step_weight_kv_bytes(cfg, len(live), live)[1])
            ctx.append(float(np.mean(live)) if live else 0.0)
            f, em = sched.step()
            forced[i] = f
            pre.append(restart)
            comp.append(bool((em > 0).any() and sched.done[em > 0].any()))
            toks.append(int(em.sum()))
        lens = [4 + int(sched.t[b]) - 1 for b in range(Bn)]
        dev_forced = torch.as_tensor(forced).cuda()
        return dict(forced=forced, dev=dev_forced, pre=pre, comp=comp, toks=toks, lens=lens, kv=kv,
                    ctx=ctx)

    def execute(pl, lo, hi, e2e=False, pin=None):
        launches = 0
        for i in range(lo, hi):
            if pl["pre"][i]:
                launches += restart_job()
            if e2e:
                pin["in"].copy_(torch.as_tensor(pl["forced"][i]))
                pin["dev_in"].copy_(pin["in"], non_blocking=True)
                B.wf_step(sess.h, None, pin["dev_in"], None, sess.out_tokens, sess.out_count, stream)
                launches += B.wf_last_launch_count(sess.h)
                pin["out_tok"].copy_(sess.out_tokens, non_blocking=True)
                pin["out_cnt"].copy_(sess.out_count, non_blocking=True)
                stream.synchronize()
            else:
                B.wf_step(sess.h, None, pl["dev"][i], None, sess.out_tokens, sess.out_count, stream)
                launches += B.wf_last_launch_count(sess.h)
            if pl["comp"][i]:
                B.wf_compact(sess.h, stream)
                launches += 1
        return launches

    local = int(os.environ.get("LOCAL_RANK", "0"))
    sampler, clock_path = _clock_sampler(_device_uuid(local))

    # ---- warm-up and the device-timed region (inputs already in HBM)
    pl = make_plan(n_steps)
    restart_job()
    execute(pl, 0, warmup)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if args.profile_region:
        torch.cuda.profiler.start()
    e0.record(stream)
    launches = execute(pl, warmup, n_steps)
    e1.record(stream)
    torch.cuda.synchronize()
    if args.profile_region:
        torch.cuda.profiler.stop()
    if world > 1:
        dist.barrier()
    dev_ms = e0.elapsed_time(e1)
    if sampler is not None:
        sampler.terminate()
        sampler.wait()
    clocks = _clock_summary(clock_path)
    try:
        os.unlink(clock_path)
    except OSError:
        pass
    tokens = sum(pl["toks"][warmup:])
    state = sess.state()
    err = sess.error()
    consistent = bool(all(int(state["len"][b]) == pl["lens"][b] for b in range(Bn)) and err == 0)

    e2e_s = e2e_tokens = None
    if e2e:
        # end to end through the C ABI: pinned host proposals in, tokens out
        Kc = cfg.block_k
        pin = {"in": torch.empty((Bn, Kc), dtype=torch.int32).pin_memory(),
               "dev_in": torch.empty((Bn, Kc), dtype=torch.int32, device="cuda"),
               "out_tok": torch.empty((Bn, Kc + 1), dtype=torch.int32).pin_memory(),
               "out_cnt": torch.empty((Bn,), dtype=torch.int32).pin_memory()}
        pl2 = make_plan(n_steps)
        restart_job()
        execute(pl2, 0, warmup)
        torch.cuda.synchronize()
        w0 = time.perf_counter()
        execute(pl2, warmup, n_steps, e2e=True, pin=pin)
        torch.cuda.synchronize()
        e2e_s = time.perf_counter() - w0
        e2e_tokens = sum(pl2["toks"][warmup:])

    # ---- per-family kernel time with CUDA events (shares of the step)
    n_prof = min(steps, 5)
    pl3 = make_plan(n_prof)
    restart_job()
    B.wf_set_option(sess.h, B.WF_OPT_PROFILE, 1)
    execute(pl3, 0, n_prof)
    prof = B.wf_profile_read(sess.h, stream)
    B.wf_set_option(sess.h, B.WF_OPT_PROFILE, 0)
    sess.close()
    del sess
    torch.cuda.empty_cache()

    wbytes = step_weight_kv_bytes(cfg, 0, [])[0]
    return dict(cfg=cfg, batch=Bn, dev_ms=dev_ms, tokens=tokens, e2e_s=e2e_s, e2e_tokens=e2e_tokens,
                prof=prof, n_prof=n_prof, clocks=clocks, consistent=consistent, err=err,
                launches=launches, wbytes=wbytes, kvbytes=float(np.mean(pl["kv"][warmup:])),
                ctx=(min(pl["ctx"][warmup:]), float(np.mean(pl["ctx"][warmup:])), max(pl["ctx"][warmup:])),
                budgets=budgets, acc=acc, enc=enc, prompt=prompt, proj_path=proj_path)


def _step_roofline(m, step_ms, hbm_peak, peak_src):
    b = m["wbytes"] + m["kvbytes"]
    return {"bytes": b, "weights": m["wbytes"], "kv": m["kvbytes"],
            "achieved_gbs": b / (step_ms * 1e-3) / 1e9, "peak_gbs": hbm_peak,
            "frac": b / (step_ms * 1e-3) / 1e9 / hbm_peak,
            "peak_source": f"{peak_src} (MEASURED_PEAKS hbm_gbs)"}


def run_ours(args, rank, world):
    import torch
    from paper_2609_32869_gb300.session import upload_weights

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    wl = WORKLOADS[args.workload]
    cfg = _cfg(wl["cfg"], wl.get("layers"))
    host_ws = syn.make_weights(cfg, seed=0)
    dev = upload_weights(host_ws)
    need_cpu = rank == 0 and world == 1 and not args.no_cpu_baseline
    m = measure_greedy(args, args.workload, dev, host_ws, rank, world, args.steps, args.warmup)
    (dev_ms, e2e_s), (tokens, e2e_tokens) = aggregate_ranks([m["dev_ms"], m["e2e_s"]],
                                                            [m["tokens"], m["e2e_tokens"]], world, "cuda")
    hbm_peak, bf16_peak, peak_src = _peaks()
    step_ms = dev_ms / args.steps
    prof, n_prof = m["prof"], m["n_prof"]
    fam = max(("gemm", "head", "attn_cross", "attn_self", "persist"), key=lambda f: prof[f]["ms"])
    roof_fam = "persist" if args.persist else "gemm"
    kernel = ("persist_kernel (every block of a pass in one launch; bytes = weights and acoustic K/V)"
              if args.persist else _proj_kernel(m["proj_path"], m["batch"] * (cfg.block_k + 1)))
    Bn, Kc = m["batch"], cfg.block_k
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
                   "block": Kc + 1, "parallelism": f"replicas x{world}",
                   "path": "persistent passes" if args.persist else "launch by launch",
                   "projections": m["proj_path"],
                   "l2": "inputs larger than L2 (every step streams "
                         f"{(m['wbytes'] + m['kvbytes']) / 1e9:.2f} GB of weights and K/V > 129 MB L2)"},
        "step_us": step_ms * 1e3,
        "tokens_per_step": tokens / args.steps / world,
        "context_len": {"min": m["ctx"][0], "mean": m["ctx"][1], "max": m["ctx"][2]},
        "step_roofline": _step_roofline(m, step_ms, hbm_peak, peak_src),
        "roofline": _family_roofline(prof, n_prof, step_ms, roof_fam, hbm_peak, peak_src, kernel,
                                     None if args.persist else _gemm_traffic(args.workload, m["proj_path"])),
        "kernel_families_ms_per_step": {k: v["ms"] / n_prof for k, v in prof.items()},
        "kernel_families_launches_per_step": {k: v["launches"] / n_prof for k, v in prof.items()},
        "top_family": fam,
        "e2e": {"value": e2e_tokens / e2e_s, "unit": "tokens/s",
                "h2d_bytes_per_step": Bn * Kc * 4,
                "d2h_bytes_per_step": Bn * (Kc + 1) * 4 + Bn * 4},
        "gpu_launches": m["launches"],
        "clocks": m["clocks"],
        "consistent": m["consistent"],
        "device_error": m["err"],
    }
    if args.workload == "large_b1" and not args.no_per_batch and not args.budget and not args.persist:
        # the metric's other batch sizes, timed in the same run on the same
        # weights (launch by launch: the persistent passes serve <= 16 rows)
        per = {}
        for name in ("large_b16", "large_b96"):
            mb = measure_greedy(args, name, dev, None, rank, world, args.batch_steps, args.warmup, e2e=False)
            (bms,), (btok,) = aggregate_ranks([mb["dev_ms"]], [mb["tokens"]], world, "cuda")
            sms = bms / args.batch_steps
            per[str(mb["batch"])] = {
                "workload": name, "description": WORKLOADS[name]["text"],
                "value": btok / (bms * 1e-3), "unit": "tokens/s", "ms_per_step": sms,
                "steps": args.batch_steps, "tokens_per_step": btok / args.batch_steps / world,
                "context_len": {"min": mb["ctx"][0], "mean": mb["ctx"][1], "max": mb["ctx"][2]},
                "step_roofline": _step_roofline(mb, sms, hbm_peak, peak_src),
                "projections": mb["proj_path"],
                "roofline": _family_roofline(mb["prof"], mb["n_prof"], sms, "gemm", hbm_peak, peak_src,
                                             _proj_kernel(mb["proj_path"], mb["batch"] * (cfg.block_k + 1)),
                                             _gemm_traffic(name, mb["proj_path"])),
                "kernel_families_ms_per_step": {k: v["ms"] / mb["n_prof"] for k, v in mb["prof"].items()},
                "clocks": mb["clocks"], "consistent": mb["consistent"], "device_error": mb["err"],
                "gpu_launches": mb["launches"]}
            if name in TENSOR_PIPE_FROM_PROFILE:
                per[str(mb["batch"])]["projection_tensor_pipe"] = TENSOR_PIPE_FROM_PROFILE[name]
        result["per_batch"] = per
    if need_cpu:
        result["cpu_baseline"] = cpu_baseline(cfg, host_ws, m["enc"], m["prompt"], m["budgets"], m["acc"],
                                              budget_s=args.cpu_seconds, gpu_ctx=m["ctx"])
    return result


def run_sampling(args, rank, world):
    """Speculative sampling steps at temperature T with the workload's proposal
    recipe: drafts sampled from q = softmax((z + sigma eps) / T), z the target's
    logits along its own sampled path (a plain-sampling pre-pass on the GPU,
    untimed) and eps seeded N(0, 1); the candidates and the logits of q go to
    wf_step, whose rejection rule takes q from them.  The job is first run
    once untimed with host reads between steps (the proposals of each step
    depend on how many tokens each sequence has emitted), recording every
    step's inputs; the timed region replays the same inputs from the same
    post-prefill state, so it runs the identical trajectory with no host
    reads.  tokens/s counts what the steps emit."""
    import torch
    import torch.distributed as dist
    from paper_2609_32869_gb300 import binding as B
    from paper_2609_32869_gb300.session import Session, upload_weights

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    wl = WORKLOADS[args.workload]
    cfg = _cfg(wl["cfg"], wl.get("layers"))
    Bn, Kc, V = wl["batch"], cfg.block_k, cfg.vocab
    T, sigma = wl["temperature"], wl["sigma"]
    dev = upload_weights(syn.make_weights(cfg, seed=0))
    enc = syn.encoder_output(cfg, Bn, seed=1)
    prompt = syn.prompts(cfg, Bn, length=4, seed=1)
    lo, hi = wl["budget"]
    budgets = syn.budgets(Bn, lo, hi, seed=2)
    sess = Session(cfg, dev, max_batch=Bn, max_ctx=cfg.max_pos)
    stream = sess.stream
    slots = np.arange(Bn, dtype=np.int32)
    d_slots = torch.as_tensor(slots, device="cuda")
    sp = B.sample_params(T, 4 + rank)
    sess.prefill(slots, enc, prompt, budgets, sp=sp)

    # pre-pass: plain sampling of the target along its own path; z[b, i] are
    # the logits the target's token i + 1 of sequence b is drawn from
    B.wf_set_option(sess.h, B.WF_OPT_KEEP_LOGITS, 1)
    z = torch.zeros((Bn, hi + Kc, V), dtype=torch.float32, device="cuda")
    pos = np.zeros(Bn, np.int64)
    sess.compact()
    while True:
        st = sess.state()
        act = [b for b in range(Bn) if not st["done"][b]]
        if not act:
            break
        sess.greedy_step(sp=sp)
        rows = sess.view(B.WF_VIEW_TARGET_LOGITS, torch.float32, (len(act), V))
        for i, b in enumerate(act):
            z[b, pos[b]] = rows[i]
            pos[b] += 1
        if any(sess.state()["done"][b] for b in act):
            sess.compact()
    B.wf_set_option(sess.h, B.WF_OPT_KEEP_LOGITS, 0)

    def restart():
        B.wf_reset_slots(sess.h, Bn, d_slots, stream)
        return B.wf_compact(sess.h, stream)

    n_steps = args.warmup + args.steps
    gen = torch.Generator(device="cuda")
    counts = torch.zeros(n_steps, Bn, dtype=torch.int32, device="cuda")
    toks = torch.zeros(n_steps, Bn, Kc + 1, dtype=torch.int32, device="cuda")
    rec_f, rec_q, rec_pre, rec_comp = [], [], [], []
    # recording pass (untimed): the proposals of each step from the emitted counts so far
    restart()
    for i in range(n_steps):
        st = sess.state()
        pre = bool((st["done"] != 0).all())
        if pre:
            restart()
            st = sess.state()
        t = np.array([int(budgets[b]) - int(st["remaining"][b]) for b in range(Bn)])
        idx = torch.as_tensor(np.clip(t[:, None] - 1 + np.arange(Kc)[None, :], 0, hi + Kc - 1),
                              device="cuda")
        gen.manual_seed(1000 + i)
        zq = torch.gather(z, 1, idx[:, :, None].expand(Bn, Kc, V)) + \
            sigma * torch.randn((Bn, Kc, V), generator=gen, device="cuda")
        u = torch.rand((Bn, Kc, V), generator=gen, device="cuda").clamp_(1e-12, 1.0)
        cand = torch.argmax(zq / T - torch.log(-torch.log(u)), dim=-1).to(torch.int32)
        B.wf_step(sess.h, sp, cand, zq, toks[i], counts[i], stream)
        done = sess.state()["done"] != 0
        comp = bool(done.any())
        if comp:
            B.wf_compact(sess.h, stream)
        rec_f.append(cand)
        rec_q.append(zq)
        rec_pre.append(pre)
        rec_comp.append(comp)
    want = counts.clone()

    def run(lo, hi_):
        n = 0
        for i in range(lo, hi_):
            if rec_pre[i]:
                restart()
                n += 2
            B.wf_step(sess.h, sp, rec_f[i], rec_q[i], toks[i], counts[i], stream)
            n += B.wf_last_launch_count(sess.h)
            if rec_comp[i]:
                B.wf_compact(sess.h, stream)
                n += 1
        return n

    sampler, clock_path = _clock_sampler(_device_uuid(local))
    restart()
    run(0, args.warmup)
    torch.cuda.synchronize()
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
    if sampler is not None:
        sampler.terminate()
        sampler.wait()
    clocks = _clock_summary(clock_path)
    try:
        os.unlink(clock_path)
    except OSError:
        pass
    c = counts[args.warmup:].cpu().numpy()
    replayed = bool(torch.equal(counts, want))
    tokens = float(c.sum())
    live = c > 0
    accepted = float((c[live] - 1).mean()) if live.any() else 0.0

    # end to end: the same replay with each step's outputs read back to pinned host memory
    h_tok = torch.empty((Bn, Kc + 1), dtype=torch.int32).pin_memory()
    h_cnt = torch.empty((Bn,), dtype=torch.int32).pin_memory()
    restart()
    run(0, args.warmup)
    torch.cuda.synchronize()
    e2e_tokens = 0
    w0 = time.perf_counter()
    for i in range(args.warmup, n_steps):
        if rec_pre[i]:
            restart()
        B.wf_step(sess.h, sp, rec_f[i], rec_q[i], toks[i], counts[i], stream)
        h_tok.copy_(toks[i], non_blocking=True)
        h_cnt.copy_(counts[i], non_blocking=True)
        stream.synchronize()
        e2e_tokens += int(h_cnt.sum())
        if rec_comp[i]:
            B.wf_compact(sess.h, stream)
    e2e_s = time.perf_counter() - w0

    n_prof = min(args.steps, 3)
    restart()
    B.wf_set_option(sess.h, B.WF_OPT_PROFILE, 1)
    run(0, n_prof)
    prof = B.wf_profile_read(sess.h, stream)
    B.wf_set_option(sess.h, B.WF_OPT_PROFILE, 0)
    st = sess.state()
    err = sess.error()
    sess.close()

    (dev_ms, e2e_s), (tokens, e2e_tokens) = aggregate_ranks([dev_ms, e2e_s], [tokens, e2e_tokens], world, "cuda")
    hbm_peak, _, peak_src = _peaks()
    step_ms = dev_ms / args.steps
    mean_L = [4 + int(budgets[b]) // 2 for b in range(Bn)]
    wbytes, kvbytes = step_weight_kv_bytes(cfg, Bn, mean_L)
    m = {"wbytes": wbytes, "kvbytes": kvbytes}
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
        "data": "synthetic (seeded random weights and encoder outputs; proposals drawn from a "
                "seeded softmax over perturbed target logits along the target's own sampled path)",
        "config": {"workload": args.workload, "description": wl["text"], "batch": Bn,
                   "block": Kc + 1, "temperature": T, "sigma": sigma,
                   "parallelism": f"replicas x{world}",
                   "l2": "inputs larger than L2 (every step streams "
                         f"{(wbytes + kvbytes) / 1e9:.2f} GB of weights and K/V > 129 MB L2)"},
        "step_us": step_ms * 1e3,
        "tokens_per_step": tokens / args.steps / world,
        "accepted_drafts_per_sequence_step": accepted,
        "acceptance_rate": accepted / Kc,
        "replayed_identically": replayed,
        "step_roofline": _step_roofline(m, step_ms, hbm_peak, peak_src),
        "roofline": _family_roofline(prof, n_prof, step_ms, "gemm", hbm_peak, peak_src,
                                     _proj_kernel("skinny" if Bn * (Kc + 1) <= 14 else "tcgen05", Bn * (Kc + 1)),
                                     None),
        "kernel_families_ms_per_step": {k: v["ms"] / n_prof for k, v in prof.items()},
        "e2e": {"value": e2e_tokens / e2e_s, "unit": "tokens/s",
                "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": Bn * (Kc + 1) * 4 + Bn * 4,
                "note": "the proposals and their logits are prepared on the device before the region"},
        "gpu_launches": launches,
        "clocks": clocks,
        "device_error": err,
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


def cpu_baseline(cfg, ws, enc, prompt, budgets, acc, budget_s=15.0, gpu_ctx=None):
    tokens, secs, steps = _oracle_run(cfg, ws, enc, prompt, budgets, acc, 0, 64,
                                      prefix_tokens=24, time_cap_s=budget_s)
    ctx = (f"; the GPU arm's steps run at context lengths {gpu_ctx[0]:.0f}..{gpu_ctx[2]:.0f} "
           f"(mean {gpu_ctx[1]:.0f}); the oracle's cost is dominated by the weights, which do not "
           f"depend on the context") if gpu_ctx else ""
    return {"value": tokens / secs, "unit": "tokens/s", "cores": _cores(), "kind": "oracle",
            "sample": f"{steps} teacher-forced speculative steps of sequence 0 over the first "
                      f"24 tokens of its transcript, context lengths 5..28 (float64 numpy oracle; "
                      f"prefill and the oracle's own greedy prefix untimed), {tokens} tokens in "
                      f"{secs:.1f} s" + ctx,
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
    ap.add_argument("--no-skinny", action="store_true",
                    help="single-sequence handles use the tcgen05 projections (WF_OPT_SKINNY 0)")
    ap.add_argument("--skinny", action="store_true",
                    help="handles of up to 144 step rows use the batched skinny projections "
                         "(WF_OPT_SKINNY 1; the default there is tcgen05)")
    ap.add_argument("--no-per-batch", action="store_true",
                    help="skip the batch-16 and batch-96 entries of the default line")
    ap.add_argument("--batch-steps", type=int, default=20,
                    help="timed steps of each per-batch entry")
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
