#!/usr/bin/env python3
"""Benchmark of the CDSL lookahead step on the 7B-shaped workload (one JSON line on rank 0).

A step is one cdsl_step: d draft decode calls over the k beams, one target verify pass over
the k*(d+1) rows, the fused epilogue, the decision and the KV commit. The metric is tokens
emitted per second (all prompts, all ranks); inputs are resident in HBM when the timed region
starts. Weights are random-init (synthetic; no checkpoints exist here), prompts are Zipf(1.1)
token ids, keywords uniform ids.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl cdsl|reference]
Multi-GPU (torchrun): every rank runs an independent replica of the workload (the prompts of
a batch are independent; no collective on the data path); value = total tokens / max time.
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
sys.path.insert(0, ROOT)

METRIC = "CDSL tokens/sec at 7B-shape target (k=4,d=4); verify-step us and % roofline"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["cdsl", "reference"], default="cdsl")
    ap.add_argument("--workload", default="7b-bf16")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--acceptance", choices=["hard", "speculative"], default="hard",
                    help="validation of the lookaheads by M_p (Sec. 3.2.2)")
    ap.add_argument("--step1-budget", type=int, choices=[0, 1, 2], default=0,
                    help="Alg. 1 S2/S3 Step-1 budget b (Sec. 3.2.3)")
    ap.add_argument("--decoder", choices=["cdsl", "cdlh", "cdlh-appx"], default="cdsl",
                    help="cdlh: the lookaheads come from M_p itself and no lookahead is ever "
                         "accepted (Alg. 2 CDLH on the same kernels); cdlh-appx: M_q's "
                         "lookaheads, never accepted (Alg. 2 CDLH-appx)")
    ap.add_argument("--verify-sweep", action="store_true",
                    help="time one cdsl_verify + cdsl_select per (k, d, prefix) point of the "
                         "7B-shape verify sweep instead of the step benchmark")
    ap.add_argument("--oracle-layers", type=int, default=2,
                    help="target layers the oracle sample runs (scaled to the full depth)")
    return ap.parse_args()


def workload(name):
    import synth
    return synth.WORKLOADS[name]


def config_of(wl):
    t, d = wl.target, wl.draft
    return {
        "workload": wl.name,
        "target": f"{t.n_layers}L/{t.d_model}/{t.n_heads}q-{t.n_kv_heads}kv/ffn{t.d_ffn}/V{t.vocab}",
        "draft": f"{d.n_layers}L/{d.d_model}/{d.n_heads}q-{d.n_kv_heads}kv/ffn{d.d_ffn}",
        "batch": wl.batch, "prompt_len": wl.prompt_len, "k": wl.k, "d": wl.d,
        "max_new": wl.max_new, "a_t": wl.a_t, "r_t": wl.r_t,
        "reward": "0.5*coverage+0.5*sigmoid(w.h)" if wl.reward_head else "coverage",
        "l2": f"inputs larger than L2: every step streams every projection and LM-head "
              f"weight ({streamed_weight_bytes(wl) / 1e9:.1f} GB; the embeddings are gathered)",
    }


def streamed_weight_bytes(wl):
    """Weight bytes one step reads through the projections: the target once, the draft once
    per lookahead call (every matrix but the embedding table, whose rows are gathered)."""
    def per_model(m):
        return sum(math.prod(s) for n, s in m.weight_specs() if n != "embed") * 2
    return per_model(wl.target) + wl.d * per_model(wl.draft)


def gemm_traffic_ratio():
    """DRAM traffic / algorithmic bytes of k_gemm_tc from the committed ncu summary, or None
    when the kernel sources changed since that capture."""
    import hashlib
    prof = os.path.join(ROOT, "profiles", "gemm_tc_7b_verify_layer.md")
    srcs = [os.path.join(ROOT, "paper_2412_10418_gb300", "csrc", f)
            for f in ("gemm_tc.cu", "gemm.cuh", "tc_ptx.cuh")]
    try:
        txt = open(prof).read()
        want = txt.split("source_sha256:")[1].split()[0]
        ratio = float(txt.split("traffic_over_algorithmic:")[1].split()[0])
        h = hashlib.sha256(b"".join(open(f, "rb").read() for f in srcs)).hexdigest()[:16]
        return ratio if h == want else None
    except Exception:
        return None


def peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        return None


# ------------------------------------------------------------------------------ clocks

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        try:
            self.p = subprocess.Popen(
                ["nvidia-smi", "-i", str(device_index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.p = None

    def stop(self):
        if self.p is None:
            return None
        time.sleep(0.25)
        self.p.terminate()
        try:
            self.p.wait(timeout=5)
        except Exception:
            self.p.kill()
        self.f.flush()
        rows = []
        for line in open(self.f.name):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), parts[5:9]))
            except ValueError:
                continue
        os.unlink(self.f.name)
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, r in rows for i, v in enumerate(r)
                          if v.lower().startswith("active")})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": rows[0][1],
                "reasons": reasons, "samples": len(rows)}


# ------------------------------------------------------------------------------ GPU arm

def build_engine(wl, device, acceptance="hard", decoder="cdsl", step1_budget=0):
    """The CDSL-k engine of a workload. decoder "cdlh": M_p drafts its own lookaheads and the
    reward threshold is above any reward (S1 never holds), so every step emits the one token
    of Alg. 2's CDLH (the step still runs its verify pass, which scores the beams).
    "cdlh-appx": M_q's lookaheads, thresholds above any score: every step emits the one
    CDLH-appx token c_{b*} (Alg. 2 with M_q as the lookahead model)."""
    import torch
    import synth
    import paper_2412_10418_gb300 as cdsl

    tw = synth.model_weights(wl, "target", device=device)
    cdlh = decoder == "cdlh"
    dw = tw if cdlh else synth.model_weights(wl, "draft", device=device)
    dshape = wl.target if cdlh else wl.draft
    head = torch.from_numpy(synth.reward_head(wl)).to(device) if wl.reward_head else None
    eng = cdsl.Engine(wl.target, dshape, wl.dtype,
                      [tw[n] for n, _ in wl.target.weight_specs()],
                      [dw[n] for n, _ in dshape.weight_specs()],
                      batch=wl.batch, k=wl.k, d=wl.d, max_prompt=wl.prompt_len,
                      max_new=wl.max_new, n_keywords=wl.n_keywords,
                      a_t=2.0 if decoder == "cdlh-appx" else wl.a_t,
                      r_t=2.0 if decoder != "cdsl" else wl.r_t, reward_head=head,
                      acceptance=cdsl.ACCEPT_SPECULATIVE if acceptance == "speculative"
                      else cdsl.ACCEPT_HARD, seed=1, step1_budget=step1_budget, device=device)
    return eng, tw, dw


def prefill(eng, wl):
    import torch
    import synth
    eng.prefill(torch.from_numpy(synth.prompts(wl)), [wl.prompt_len] * wl.batch,
                torch.from_numpy(synth.keywords(wl)))


def timed_steps(eng, wl, n_steps, warmup):
    """Warm up, then time n_steps cdsl_step calls (CUDA events on the engine's stream).

    The decoding state advances every step; when a prompt could reach l_m within the next
    segment, the context is re-prefilled outside the timed region, so every timed step does
    the full work and emits at least one token per prompt."""
    import torch
    per_seg = max(1, wl.max_new // (wl.d + 1))
    prefill(eng, wl)
    for _ in range(warmup):
        eng.step()
    eng.stream.synchronize()
    total_ms, tokens, done = 0.0, 0, 0
    left_in_seg = per_seg - warmup
    while done < n_steps:
        if left_in_seg <= 0:
            prefill(eng, wl)
            left_in_seg = per_seg
        n = min(left_in_seg, n_steps - done)
        c0 = eng.counters()[3]
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        eng.stream.synchronize()
        e0.record(eng.stream)
        for _ in range(n):
            eng.step()
        e1.record(eng.stream)
        eng.stream.synchronize()
        total_ms += e0.elapsed_time(e1)
        tokens += eng.counters()[3] - c0
        done += n
        left_in_seg -= n
    return total_ms, tokens


def kernel_timing(eng, wl, n_steps):
    """Per-launch CUDA events around every projection GEMM over n_steps steps (direct launches
    on the engine's stream), and the verify call alone."""
    import torch
    import paper_2412_10418_gb300 as cdsl
    prefill(eng, wl)
    eng.step()
    cdsl.cdsl_profile(eng.ctx, True)
    for _ in range(n_steps):
        eng.step()
    prof = {name: cdsl.cdsl_get_profile(eng.ctx, impl) for impl, name in cdsl.KERNEL_CLASSES.items()}
    # tensor-core GEMM launches grouped by shape (equal algorithmic bytes = same projection)
    groups = {}
    for cls, ms, by, fl in cdsl.cdsl_get_profile_launches(eng.ctx):
        if cls != 2:
            continue
        g = groups.setdefault(round(by), [0, 0.0])
        g[0] += 1
        g[1] += ms
    cdsl.cdsl_profile(eng.ctx, False)
    prof["_gemm_shapes"] = groups
    # verify-step time: lookahead, then the verify call alone between events
    ts = []
    for _ in range(n_steps):
        eng.lookahead()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(eng.stream)
        eng.verify()
        e1.record(eng.stream)
        eng.select()
        eng.stream.synchronize()
        ts.append(e0.elapsed_time(e1))
    return prof, statistics.median(ts) * 1000.0


def e2e_run(eng, wl, n_steps):
    """tokens/s through the public API with host buffers, for whole generations: pinned
    prompts and keywords are copied in, the prompts prefilled, then steps run until every
    prompt has its l_m tokens, each step's emitted tokens read back to the host."""
    import torch
    import synth
    import paper_2412_10418_gb300 as cdsl
    n_steps = wl.max_new     # at least one token per step per live prompt
    hp = torch.from_numpy(synth.prompts(wl)).pin_memory()
    hk = torch.from_numpy(synth.keywords(wl)).pin_memory()
    out_tok = torch.empty((wl.batch, wl.d + 1), dtype=torch.int32).pin_memory()
    out_n = torch.empty(wl.batch, dtype=torch.int32).pin_memory()
    dp = torch.empty(hp.shape, dtype=torch.int32, device=eng.ws.device)
    dk = torch.empty(hk.shape, dtype=torch.int32, device=eng.ws.device)
    eng.stream.synchronize()
    t0 = time.perf_counter()
    with torch.cuda.stream(eng.stream):
        dp.copy_(hp, non_blocking=True)
        dk.copy_(hk, non_blocking=True)
    cdsl.cdsl_prefill(eng.ctx, dp, [wl.prompt_len] * wl.batch, dk)
    tokens = 0
    done = 0
    for _ in range(n_steps):
        eng.step()
        with torch.cuda.stream(eng.stream):
            out_tok.copy_(eng.emitted, non_blocking=True)
            out_n.copy_(eng.n_emitted, non_blocking=True)
        eng.stream.synchronize()
        tokens += int(out_n.sum())
        done += 1
        if tokens >= wl.batch * wl.max_new:
            break
    dt = time.perf_counter() - t0
    n_steps = done
    h2d = (hp.numel() + hk.numel()) * 4 / n_steps
    d2h = (out_tok.numel() + out_n.numel()) * 4
    return tokens / dt, h2d, d2h, n_steps


# ------------------------------------------------------------------------------ oracle arm

def oracle_sample(wl, tw_host_fn, dw_host, n_layers, steps=1, warmup=0):
    """The oracle as it stands on a bounded sample of the workload: CDSL-k steps of the
    7B-shaped models over a 16-token prompt with the target cut to its first n_layers layers.
    Returns (seconds per full step, scaled to the full target depth, cores)."""
    import numpy as np
    import synth
    import oracle
    tshape = wl.target
    cut = synth.ModelShape(n_layers=n_layers, d_model=tshape.d_model, n_heads=tshape.n_heads,
                           n_kv_heads=tshape.n_kv_heads, d_ffn=tshape.d_ffn, vocab=tshape.vocab)
    tgt = oracle.Transformer(cut, tw_host_fn(n_layers), keep_widened=False)
    drf = oracle.Transformer(wl.draft, dw_host, keep_widened=True)
    for name in dw_host:          # the draft's fp64 copies are cached by the oracle after use
        drf.w(name)
    run = oracle.RunParams(k=wl.k, d=wl.d, a_t=wl.a_t, r_t=wl.r_t, max_new=10_000,
                           composite_reward=wl.reward_head)
    prompt = synth.prompts(wl)[:1, :16]
    states = oracle.prefill(tgt, drf, prompt, synth.keywords(wl)[:1])
    w = synth.reward_head(wl)
    for _ in range(warmup):
        oracle.cdsl_k_step(tgt, drf, states, run, w)
    t_draft = t_tgt = 0.0
    for _ in range(steps):
        # the same step split into its two model parts, to scale the target part
        t0 = time.perf_counter()
        dcs = [states[0].dcache.fork() for _ in range(wl.k)]
        roots = np.argsort(-states[0].p_root)[:wl.k].tolist()
        feed = roots
        xs = [[] for _ in range(wl.k)]
        for j in range(wl.d):
            lg, _ = drf.forward([(dcs[i], [feed[i]]) for i in range(wl.k)])
            feed = [int(np.argmax(l[0])) for l in lg]
            for i in range(wl.k):
                xs[i].append(feed[i])
        t1 = time.perf_counter()
        tgt.forward([(states[0].tcache.fork(), [roots[i]] + xs[i]) for i in range(wl.k)])
        t2 = time.perf_counter()
        t_draft += t1 - t0
        t_tgt += t2 - t1
    per_layer = t_tgt / steps / n_layers
    step_s = t_draft / steps + per_layer * tshape.n_layers
    return step_s, os.cpu_count()


def host_weights_fns(wl, tw, dw):
    import synth

    def target_cut(n):
        keep = {"embed", "final_norm", "lm_head"} | {f"l{l}.{x}" for l in range(n) for x in
                                                      ("attn_norm", "wq", "wk", "wv", "wo",
                                                       "ffn_norm", "w_gate", "w_up", "w_down")}
        return synth.to_host({k: v for k, v in tw.items() if k in keep})

    return target_cut, synth.to_host(dw)


def cpu_baseline(wl, tw, dw, tokens_per_step, n_layers):
    fn, dh = host_weights_fns(wl, tw, dw)
    step_s, cores = oracle_sample(wl, fn, dh, n_layers)
    return {"value": tokens_per_step * wl.batch / step_s, "unit": "tokens/s", "cores": cores,
            "kind": "oracle",
            "sample": (f"one CDSL-k step (B=1, k={wl.k}, d={wl.d}) of the fp64 oracle on a "
                       f"16-token prompt: draft {wl.d} calls x {wl.k} beams in full, target "
                       f"{n_layers} of {wl.target.n_layers} layers timed and scaled to the full "
                       f"depth; {tokens_per_step:.2f} tokens/step as measured on the GPU")}


# ------------------------------------------------------------------------------ ranks

def aggregate_ranks(total_ms, tokens, device="cpu"):
    """Whole-job numbers over the ranks of the default process group: the slowest rank's
    time and the tokens of all ranks (replicas: every rank decodes the whole workload on its
    own GPU, nothing is exchanged on the data path)."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(total_ms), float(tokens)], device=device, dtype=torch.float64)
    mx = t.clone()
    dist.all_reduce(mx, op=dist.ReduceOp.MAX)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(mx[0]), float(t[1])


def sum_over_ranks(x, device="cpu"):
    """A per-rank rate summed over the ranks (the end-to-end tokens/s of the replicas)."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], device=device, dtype=torch.float64)
    dist.all_reduce(t)
    return float(t[0])


# ------------------------------------------------------------------------------ main

def gpu_main(args):
    import torch
    import torch.distributed as dist

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    device = f"cuda:{local}"
    from paper_2412_10418_gb300 import build as b
    if rank == 0:
        b.build()
    if world > 1:
        dist.barrier()
    wl = workload(args.workload)
    eng, tw, dw = build_engine(wl, device, args.acceptance, args.decoder, args.step1_budget)

    if world > 1:
        dist.barrier()
    clocks = ClockSampler(local)
    total_ms, tokens = timed_steps(eng, wl, args.steps, args.warmup)
    clk = clocks.stop()
    if world > 1:
        total_ms, tokens = aggregate_ranks(total_ms, tokens, device)
    value = tokens / (total_ms / 1000.0)
    counters = eng.counters()
    launches_per_step = counters[6]

    n_prof = min(args.steps, 5)
    prof, verify_us = kernel_timing(eng, wl, n_prof)
    shapes = prof.pop("_gemm_shapes")
    import paper_2412_10418_gb300 as cdsl
    gem = {k: v for k, v in prof.items() if k in cdsl.GEMM_IMPLS.values()}
    dom = max(gem.items(), key=lambda kv: kv[1]["ms"])
    pk = peaks()
    hbm = pk["hbm_gbs"] if pk else 6800.0
    achieved = dom[1]["bytes"] / (dom[1]["ms"] / 1000.0) / 1e9 if dom[1]["ms"] > 0 else 0.0
    ratio = gemm_traffic_ratio() if dom[0] == "gemm_tc" else None
    bpl = dom[1]["bytes"] / max(1, dom[1]["launches"])
    roofline = {"bound": "hbm", "kernel": dom[0], "achieved": round(achieved, 1),
                "peak": hbm, "unit": "GB/s", "frac": round(achieved / hbm, 4),
                "traffic": round(ratio * bpl) if ratio else None,
                "peak_source": "measured" if pk else "fallback",
                "timing": "CUDA events around each launch, direct launches (no graph overlap)",
                "launches_timed": dom[1]["launches"],
                "avg_launch_us": round(dom[1]["ms"] * 1000.0 / max(1, dom[1]["launches"]), 2),
                "bytes_per_launch": round(dom[1]["bytes"] / max(1, dom[1]["launches"]))}
    # per projection shape (the same kernel, different launch shapes): the largest by time
    by_shape = sorted(({"bytes_per_launch": b, "launches": n, "avg_us": round(ms * 1000.0 / n, 2),
                        "GB/s": round(b / (ms / n / 1000.0) / 1e9, 1),
                        "frac": round(b / (ms / n / 1000.0) / 1e9 / hbm, 3)}
                       for b, (n, ms) in shapes.items()), key=lambda r: -r["avg_us"] * r["launches"])
    roofline["by_shape"] = by_shape[:8]
    # the same bytes over the graph-replayed step (everything else in the step included): a
    # lower bound on the projections' rate inside the CUDA graph
    step_bytes = dom[1]["bytes"] / n_prof
    step_ms = total_ms / args.steps   # every rank times args.steps steps; the slowest rank
    roofline["in_graph_lower_bound"] = {
        "bytes_per_step": round(step_bytes), "ms_per_step": round(step_ms, 4),
        "GB/s": round(step_bytes / (step_ms / 1000.0) / 1e9, 1),
        "frac": round(step_bytes / (step_ms / 1000.0) / 1e9 / hbm, 4)}
    verify_bytes = (wl.target.n_params() * 2)
    e2e = None
    if not args.no_e2e:
        ev, h2d, d2h, n_e2e = e2e_run(eng, wl, args.steps)
        if world > 1:
            ev = sum_over_ranks(ev, device)
        e2e = {"value": round(ev, 3), "unit": "tokens/s", "h2d_bytes_per_step": round(h2d, 1),
               "d2h_bytes_per_step": d2h,
               "note": f"whole generations: pinned prompts+keywords in, prefill, then {n_e2e} "
                       "cdsl_step calls (until every prompt has max_new tokens), each "
                       "followed by a read of the emitted tokens"}
    out = None
    if rank == 0:
        tokens_per_step = tokens / (args.steps * max(1, world)) / wl.batch
        cpu = None
        if not args.no_cpu_baseline and world == 1 and args.decoder == "cdsl":
            cpu = cpu_baseline(wl, tw, dw, tokens_per_step, args.oracle_layers)
        out = {
            "metric": METRIC, "value": round(value, 3), "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(total_ms / args.steps, 4), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": dict(config_of(wl), parallelism=f"replicas{world}",
                           acceptance=args.acceptance, decoder=args.decoder,
                           step1_budget=args.step1_budget,
                           **({"draft": "= target (CDLH)", "r_t": None}
                              if args.decoder == "cdlh" else {}),
                           **({"a_t": None, "r_t": None} if args.decoder == "cdlh-appx" else {})),
            "verify_us": round(verify_us, 1),
            "verify_gbs": round(verify_bytes / (verify_us * 1e-6) / 1e9, 1),
            "tokens_per_step": round(tokens_per_step, 3),
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "clocks": clk,
            "gpu_launches": int(launches_per_step * args.steps),
            "kernel_profile": {k: {"launches": v["launches"], "ms_per_step": round(v["ms"] / n_prof, 3),
                                   "GB/s": round(v["bytes"] / (v["ms"] / 1e3) / 1e9, 1) if v["bytes"] else None}
                               for k, v in prof.items() if v["launches"]},
        }
        print(json.dumps(out), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()
    eng.close()


def reference_main(args):
    """The oracle arm: the fp64 oracle as it stands on the host cores, each step a bounded
    sample of the same workload (rank 0 only; other ranks exit without work)."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import torch
    wl = workload(args.workload)
    device = "cuda:0" if torch.cuda.is_available() else "cpu"
    import synth
    # weights drawn exactly as the GPU arm draws them, then copied to the host
    tw = synth.model_weights(wl, "target", device=device)
    dw = synth.model_weights(wl, "draft", device=device)
    fn, dh = host_weights_fns(wl, tw, dw)
    del tw, dw
    step_s, cores = oracle_sample(wl, fn, dh, args.oracle_layers, steps=args.steps,
                                  warmup=args.warmup)
    value = wl.batch / step_s   # one token per prompt and step (the GPU arm's measured rate)
    sample = (f"per step: one CDSL-k step (B=1, k={wl.k}, d={wl.d}) of the fp64 oracle on a "
              f"16-token prompt, target {args.oracle_layers} of {wl.target.n_layers} layers "
              "timed and scaled to the full depth; 1 token per step")
    out = {"metric": METRIC, "value": round(value, 6), "unit": "tokens/s", "n_gpus": 1,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(step_s * 1e3, 1),
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": "synthetic", "impl": "reference", "config": config_of(wl),
           "cpu_baseline": {"value": round(value, 6), "unit": "tokens/s", "kind": "oracle",
                            "cores": cores, "sample": sample},
           "e2e": {"value": round(value, 6), "unit": "tokens/s", "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def verify_sweep(args):
    """The verify-kernel sweep on the 7B-shape target: for k in {2,4,8,16}, d in {2,...,10},
    prefix in {512,...,4096}, one cdsl_verify + cdsl_select call (after an untimed lookahead)
    timed with CUDA events on the engine's stream (median of 3 after 1 warm-up), next to k*d
    sequential target decode steps (the k=1, d=1 verify of the same prefix, 2 rows, stands in
    for one decode step). One JSON line per point."""
    import torch
    import synth
    import paper_2412_10418_gb300 as cdsl
    from paper_2412_10418_gb300 import build as b
    b.build()
    wl0 = workload("7b-bf16")
    tw = synth.model_weights(wl0, "target", device="cuda")
    dw = synth.model_weights(wl0, "draft", device="cuda")
    head = torch.from_numpy(synth.reward_head(wl0)).cuda()
    wbytes = wl0.target.n_params() * 2
    pk = peaks()
    hbm = pk["hbm_gbs"] if pk else 6800.0
    tfl = pk.get("bf16_tflops") if pk else None

    def time_point(k, d, prefix, reps=3):
        wl = synth.scaled(wl0, k=k, d=d, prompt_len=prefix, max_new=4 * reps + 8)
        eng = cdsl.Engine(wl.target, wl.draft, wl.dtype,
                          [tw[n] for n, _ in wl.target.weight_specs()],
                          [dw[n] for n, _ in wl.draft.weight_specs()], batch=1, k=k, d=d,
                          max_prompt=prefix, max_new=wl.max_new, n_keywords=wl.n_keywords,
                          a_t=wl.a_t, r_t=wl.r_t, reward_head=head, device="cuda")
        prefill(eng, wl)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ts = []
        for r in range(reps + 1):
            eng.lookahead()
            eng.stream.synchronize()
            e0.record(eng.stream)
            eng.verify()
            eng.select()
            e1.record(eng.stream)
            e1.synchronize()
            if r:
                ts.append(e0.elapsed_time(e1) * 1000.0)
        eng.close()
        return sorted(ts)[len(ts) // 2]

    for prefix in (512, 1024, 2048, 4096):
        t_dec = time_point(1, 1, prefix)
        for k in (2, 4, 8, 16):
            for d in (2, 4, 6, 8, 10):
                us = time_point(k, d, prefix)
                rows = k * (d + 1)
                flops = 2.0 * wl0.target.n_params() * rows
                out = {"sweep": "verify", "k": k, "d": d, "prefix": prefix, "rows": rows,
                       "verify_select_us": round(us, 1),
                       "weights_gbs": round(wbytes / (us * 1e-6) / 1e9, 1),
                       "hbm_frac": round(wbytes / (us * 1e-6) / 1e9 / hbm, 3),
                       "tflops": round(flops / (us * 1e-6) / 1e12, 2),
                       "tensor_frac": round(flops / (us * 1e-6) / 1e12 / tfl, 4) if tfl else None,
                       "decode_step_us": round(t_dec, 1),
                       "sequential_kd_decode_us": round(k * d * t_dec, 1),
                       "speedup_vs_sequential": round(k * d * t_dec / us, 2)}
                print(json.dumps(out), flush=True)


if __name__ == "__main__":
    a = parse()
    if a.impl == "reference":
        reference_main(a)
    elif a.verify_sweep:
        verify_sweep(a)
    else:
        gpu_main(a)
