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
    ap.add_argument("--sweep-k", default="2,4,8,16", help="verify sweep: beam counts k")
    ap.add_argument("--sweep-d", default="2,4,6,8,10", help="verify sweep: lookahead lengths d")
    ap.add_argument("--sweep-prefix", default="512,1024,2048,4096",
                    help="verify sweep: prefix lengths")
    ap.add_argument("--oracle-layers", type=int, default=2,
                    help="target layers the oracle sample runs (scaled to the full depth)")
    ap.add_argument("--draft-equals-target", action="store_true",
                    help="forced acceptance: the draft is the target model itself, so every "
                         "lookahead is accepted and S1 steps emit several tokens")
    ap.add_argument("--oracle-worker", default=None, help=argparse.SUPPRESS)
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


def streamed_weight_bytes_model(m):
    """Weight bytes one forward pass of a bf16 model streams: every matrix but the embedding
    table, whose rows are only gathered."""
    return sum(math.prod(s) for n, s in m.weight_specs() if n != "embed") * 2


def streamed_weight_bytes(wl):
    """Weight bytes one step reads through the projections: the target once, the draft once
    per lookahead call."""
    return streamed_weight_bytes_model(wl.target) + wl.d * streamed_weight_bytes_model(wl.draft)


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

def build_engine(wl, device, acceptance="hard", decoder="cdsl", step1_budget=0,
                 draft_equals_target=False):
    """The CDSL-k engine of a workload. decoder "cdlh": M_p drafts its own lookaheads and the
    reward threshold is above any reward (S1 never holds), so every step emits the one token
    of Alg. 2's CDLH (the step still runs its verify pass, which scores the beams).
    "cdlh-appx": M_q's lookaheads, thresholds above any score: every step emits the one
    CDLH-appx token c_{b*} (Alg. 2 with M_q as the lookahead model).
    draft_equals_target (CDSL only): M_p drafts its own lookaheads and r_t = 0, so every
    lookahead is accepted and every step is S1, emitting c_b* and all d drafts (the forced
    acceptance diagnostic of the S1 path: multi-token emission, multi-row KV commit, the
    pending draft row of the next step)."""
    import torch
    import synth
    import paper_2412_10418_gb300 as cdsl

    tw = synth.model_weights(wl, "target", device=device)
    cdlh = decoder == "cdlh" or draft_equals_target
    dw = tw if cdlh else synth.model_weights(wl, "draft", device=device)
    dshape = wl.target if cdlh else wl.draft
    r_t = 0.0 if draft_equals_target else (2.0 if decoder != "cdsl" else wl.r_t)
    head = torch.from_numpy(synth.reward_head(wl)).to(device) if wl.reward_head else None
    eng = cdsl.Engine(wl.target, dshape, wl.dtype,
                      [tw[n] for n, _ in wl.target.weight_specs()],
                      [dw[n] for n, _ in dshape.weight_specs()],
                      batch=wl.batch, k=wl.k, d=wl.d, max_prompt=wl.prompt_len,
                      max_new=wl.max_new, n_keywords=wl.n_keywords,
                      a_t=2.0 if decoder == "cdlh-appx" else wl.a_t,
                      r_t=r_t, reward_head=head,
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
    """Kernel classes inside the graph-replayed step (cdsl_profile mode 2: the kernels stamp
    their first block's entry and last block's exit; each launch is charged the part of its
    interval after the previous stamped exit, so the charged times never add up to more than
    the step), the same launches bracketed by CUDA events outside the graph (mode 1), and the
    verify call alone between events."""
    import torch
    import paper_2412_10418_gb300 as cdsl
    prefill(eng, wl)
    eng.step()

    def read(mode):
        prof = {name: cdsl.cdsl_get_profile(eng.ctx, impl)
                for impl, name in cdsl.KERNEL_CLASSES.items()}
        launches = cdsl.cdsl_get_profile_launches(eng.ctx)
        if mode == cdsl.PROFILE_IN_GRAPH:
            prof["_steps"] = cdsl.cdsl_get_profile(eng.ctx, cdsl.STAMPED_STEPS)
        cdsl.cdsl_profile(eng.ctx, cdsl.PROFILE_OFF)
        return prof, launches

    cdsl.cdsl_profile(eng.ctx, cdsl.PROFILE_IN_GRAPH)
    for _ in range(n_steps):
        eng.step()
    in_graph = read(cdsl.PROFILE_IN_GRAPH)
    cdsl.cdsl_profile(eng.ctx, cdsl.PROFILE_EVENTS)
    for _ in range(n_steps):
        eng.step()
    events = read(cdsl.PROFILE_EVENTS)
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
    return in_graph, events, statistics.median(ts) * 1000.0


def by_shape(launches, cls, per_step_div, hbm):
    """Launches of one class grouped by algorithmic bytes (one group per projection shape),
    largest total time first. In mode 2 a launch record's milliseconds are already per step;
    in mode 1 they are per launch (per_step_div = steps profiled)."""
    groups = {}
    for c, ms, by, fl in launches:
        if c != cls or by <= 0:
            continue
        g = groups.setdefault(round(by), [0, 0.0])
        g[0] += 1
        g[1] += ms
    rows = []
    for b, (n, ms) in groups.items():
        if ms <= 0:
            continue
        per_launch_ms = ms / n
        gbs = b / (per_launch_ms / 1000.0) / 1e9
        rows.append({"bytes_per_launch": b, "launches_per_step": round(n / per_step_div, 2),
                     "avg_us": round(per_launch_ms * 1000.0, 2), "GB/s": round(gbs, 1),
                     "frac": round(gbs / hbm, 3)})
    return sorted(rows, key=lambda r: -r["avg_us"] * r["launches_per_step"])


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

ORACLE_PREFIX = "oracle_"


def cut_shape(shape, n_layers):
    import synth
    return synth.ModelShape(n_layers=n_layers, d_model=shape.d_model, n_heads=shape.n_heads,
                            n_kv_heads=shape.n_kv_heads, d_ffn=shape.d_ffn, vocab=shape.vocab,
                            rope_theta=shape.rope_theta, norm_eps=shape.norm_eps)


def oracle_worker(args):
    """The oracle as it stands, in a process of its own (its BLAS thread count is fixed by the
    environment the parent gives it): CDSL-k steps of the first prompt of the workload on its
    real prompt, the draft at full depth and the target cut to its first --oracle-layers
    layers (plus embedding, final norm and LM head). The first worker prefills and saves the
    decoding state; later workers start from that saved state. Prints one JSON line."""
    import pickle
    import numpy as np
    import synth
    import oracle
    wdir = args.oracle_worker
    meta = json.load(open(os.path.join(wdir, "meta.json")))
    wl = synth.WORKLOADS[meta["workload"]]
    n_cut = meta["layers"]
    def load(prefix):
        return {f[len(prefix):-4]: np.load(os.path.join(wdir, f), mmap_mode="r")
                for f in os.listdir(wdir) if f.startswith(prefix) and f.endswith(".npy")}
    tgt = oracle.Transformer(cut_shape(wl.target, n_cut), load("t_"), keep_widened=True)
    drf = oracle.Transformer(wl.draft, load("d_"), keep_widened=True)
    for m in (tgt, drf):                  # widen every matrix once, before any timing
        for name in m.raw:
            m.w(name)
    run = oracle.RunParams(k=wl.k, d=wl.d, a_t=wl.a_t, r_t=wl.r_t, max_new=10_000,
                           composite_reward=wl.reward_head)
    w_head = synth.reward_head(wl)
    st_path = os.path.join(wdir, "states.pkl")
    prefill_s = None
    if os.path.exists(st_path):
        states = pickle.load(open(st_path, "rb"))
    else:
        t0 = time.perf_counter()
        states = oracle.prefill(tgt, drf, synth.prompts(wl)[:1], synth.keywords(wl)[:1])
        prefill_s = time.perf_counter() - t0
        pickle.dump(states, open(st_path, "wb"))
    step_s, tgt_s, tokens = [], [], 0
    for i in range(meta["warmup"] + meta["steps"]):
        t0 = time.perf_counter()
        rec = oracle.cdsl_k_step(tgt, drf, states, run, w_head)[0]
        t1 = time.perf_counter()
        # the step's target pass alone (same rows, a forked cache), for the depth scaling
        tgt.forward([(states[0].tcache.fork(), [int(rec.roots[j])] + rec.x[j].tolist())
                     for j in range(wl.k)])
        t2 = time.perf_counter()
        if i >= meta["warmup"]:
            step_s.append(t1 - t0)
            tgt_s.append(t2 - t1)
            tokens += len(rec.emitted)
    print(json.dumps({"threads": int(os.environ.get("OPENBLAS_NUM_THREADS", "0") or 0),
                      "prefill_s": prefill_s, "step_s": step_s, "target_s": tgt_s,
                      "tokens": tokens}), flush=True)


def oracle_runs(wl, tw, dw, n_layers, runs):
    """Run oracle_worker processes on the host cores: runs = [(threads, warmup, steps), ...],
    the first of them also prefilling the real prompt. tw / dw: the engine's weights (torch
    tensors, any device). Returns one result dict per run, with the depth-scaled estimate of
    a full-depth step added (the target's share scaled by the streamed weights of the full
    target over those of the cut one: the verify pass's flops are proportional to them)."""
    import shutil
    import numpy as np
    import synth
    keep_t = {"embed", "final_norm", "lm_head"} | {
        f"l{l}.{x}" for l in range(n_layers)
        for x in ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate", "w_up", "w_down")}
    wdir = tempfile.mkdtemp(prefix="cdsl_oracle_")
    try:
        for prefix, src, keep in (("t_", tw, keep_t), ("d_", dw, None)):
            for name, arr in synth.to_host({k: v for k, v in src.items()
                                            if keep is None or k in keep}).items():
                np.save(os.path.join(wdir, prefix + name + ".npy"), arr)
        out = []
        for threads, warmup, steps in runs:
            json.dump({"workload": wl.name, "layers": n_layers, "warmup": warmup,
                       "steps": steps}, open(os.path.join(wdir, "meta.json"), "w"))
            env = dict(os.environ, OPENBLAS_NUM_THREADS=str(threads), OMP_NUM_THREADS=str(threads),
                       MKL_NUM_THREADS=str(threads))
            r = subprocess.run([sys.executable, os.path.abspath(__file__), "--oracle-worker", wdir],
                               env=env, capture_output=True, text=True, timeout=1800)
            if r.returncode != 0:
                raise RuntimeError(f"oracle worker ({threads} threads) failed: {r.stderr[-2000:]}")
            res = json.loads(r.stdout.strip().splitlines()[-1])
            ratio = (streamed_weight_bytes_model(wl.target) /
                     streamed_weight_bytes_model(cut_shape(wl.target, n_layers)))
            n = max(1, len(res["step_s"]))
            res["sample_step_s"] = sum(res["step_s"]) / n
            res["full_depth_step_s"] = (sum(res["step_s"]) + (ratio - 1.0) * sum(res["target_s"])) / n
            res["tokens_per_step"] = res["tokens"] / n
            out.append(res)
        return out
    finally:
        shutil.rmtree(wdir, ignore_errors=True)


def oracle_sample_text(wl, n_layers):
    return (f"CDSL-k steps of the fp64 oracle on the workload's first prompt ({wl.prompt_len} "
            f"tokens, prefilled once), k={wl.k}, d={wl.d}: the draft at its full "
            f"{wl.draft.n_layers} layers, the target cut to {n_layers} of "
            f"{wl.target.n_layers} layers; the measured step is scaled to the full target depth "
            "by the ratio of streamed target weights (the verify pass's flops follow them)")


def cpu_baseline(wl, tw, dw, n_layers):
    """The oracle timed on the host cores at all cores and at 1 thread, one step each after
    the prefill (value: all cores, full-depth estimate)."""
    cores = os.cpu_count()
    allc, one = oracle_runs(wl, tw, dw, n_layers, [(cores, 0, 1), (1, 0, 1)])
    def summary(r):
        return {"threads": r["threads"], "sample_ms_per_step": round(r["sample_step_s"] * 1e3, 1),
                "full_depth_ms_per_step_estimate": round(r["full_depth_step_s"] * 1e3, 1),
                "tokens_per_s": round(r["tokens_per_step"] / r["full_depth_step_s"], 6)}
    return {"value": round(allc["tokens_per_step"] / allc["full_depth_step_s"], 6),
            "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": oracle_sample_text(wl, n_layers),
            "prefill_s": round(allc["prefill_s"], 1) if allc["prefill_s"] else None,
            "all_cores": summary(allc), "one_thread": summary(one)}


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
    eng, tw, dw = build_engine(wl, device, args.acceptance, args.decoder, args.step1_budget,
                               args.draft_equals_target)

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
    (prof, launches), (prof_ev, launches_ev), verify_us = kernel_timing(eng, wl, n_prof)
    import paper_2412_10418_gb300 as cdsl
    pk = peaks()
    hbm = pk["hbm_gbs"] if pk else 6800.0
    step_ms = total_ms / args.steps   # every rank times args.steps steps; the slowest rank
    stamped = prof.pop("_steps")
    gem = {k: v for k, v in prof.items() if k in cdsl.GEMM_IMPLS.values()}
    dom = max(gem.items(), key=lambda kv: kv[1]["ms"])
    d = dom[1]
    n_launch = max(1, d["launches"])
    avg_ms = d["ms"] / n_launch
    bpl = d["bytes"] / n_launch
    achieved = bpl / (avg_ms / 1000.0) / 1e9 if avg_ms > 0 else 0.0
    ratio = gemm_traffic_ratio() if dom[0] == "gemm_tc" else None
    charged = sum(v["ms"] for v in prof.values()) / n_prof
    roofline = {"bound": "hbm", "kernel": dom[0], "achieved": round(achieved, 1),
                "peak": hbm, "unit": "GB/s", "frac": round(achieved / hbm, 4),
                "traffic": round(ratio * bpl) if ratio else None,
                "peak_source": "measured" if pk else "fallback",
                "timing": "in the CUDA graph: per-launch %globaltimer stamps (first block "
                          "entry, last block exit), each launch charged after the previous "
                          "stamped exit; the charged times of a step never overlap",
                "launches_per_step": round(d["launches"] / n_prof, 1),
                "avg_launch_us": round(avg_ms * 1000.0, 2),
                "bytes_per_launch": round(bpl),
                "ms_per_step_in_graph": round(d["ms"] / n_prof, 4),
                "stamped_step_ms": round(stamped["ms"] / max(1, stamped["launches"]), 4),
                "charged_ms_per_step_all_classes": round(charged, 4)}
    roofline["by_shape"] = by_shape(launches, 2, 1, hbm)[:10]
    att = prof.get("attention", {})
    if att.get("ms"):
        a_bpl = att["bytes"] / max(1, att["launches"])
        a_ms = att["ms"] / max(1, att["launches"])
        a_gbs = a_bpl / (a_ms / 1000.0) / 1e9
        roofline["attention"] = {
            "bound": "hbm", "launches_per_step": round(att["launches"] / n_prof, 1),
            "avg_launch_us": round(a_ms * 1000.0, 2), "bytes_per_launch": round(a_bpl),
            "achieved": round(a_gbs, 1), "frac": round(a_gbs / hbm, 4),
            "ms_per_step_in_graph": round(att["ms"] / n_prof, 4),
            "bytes": "counted by the kernel: K and V (fp32) of every key once per prompt and "
                     "KV head, every query vector read and its output written once",
            "by_shape": by_shape(launches, 3, 1, hbm)[:6]}
    roofline["in_graph_ms_per_step"] = {k: round(v["ms"] / n_prof, 4) for k, v in prof.items()
                                        if v["ms"] > 0}
    # the same launches bracketed by CUDA events outside the graph (no overlap between them)
    dev = prof_ev.get(dom[0], {})
    if dev.get("ms"):
        ev_ms = dev["ms"] / max(1, dev["launches"])
        ev_bpl = dev["bytes"] / max(1, dev["launches"])
        roofline["event_timed"] = {
            "timing": "CUDA events around each launch on the engine's stream, direct launches "
                      "(no graph, no programmatic overlap)",
            "avg_launch_us": round(ev_ms * 1000.0, 2),
            "achieved": round(ev_bpl / (ev_ms / 1000.0) / 1e9, 1),
            "frac": round(ev_bpl / (ev_ms / 1000.0) / 1e9 / hbm, 4),
            "by_shape": by_shape(launches_ev, 2, n_prof, hbm)[:10]}
    verify_bytes = streamed_weight_bytes_model(wl.target)
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
        if (not args.no_cpu_baseline and world == 1 and args.decoder == "cdsl"
                and not args.draft_equals_target):
            cpu = cpu_baseline(wl, tw, dw, args.oracle_layers)
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
                           **({"a_t": None, "r_t": None} if args.decoder == "cdlh-appx" else {}),
                           **({"draft": "= target (forced acceptance)", "r_t": 0.0}
                              if args.draft_equals_target else {})),
            "verify_us": round(verify_us, 1),
            "verify_gbs": round(verify_bytes / (verify_us * 1e-6) / 1e9, 1),
            "tokens_per_step": round(tokens_per_step, 3),
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "clocks": clk,
            "gpu_launches": int(launches_per_step * args.steps),
            "kernel_profile": {k: {"launches_per_step": round(v["launches"] / n_prof, 1),
                                   "ms_per_step_in_graph": round(v["ms"] / n_prof, 4),
                                   "GB/s": (round(v["bytes"] / (v["ms"] / 1e3) / 1e9, 1)
                                            if v["bytes"] and v["ms"] else None)}
                               for k, v in prof.items() if v["launches"]},
        }
        print(json.dumps(out), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()
    eng.close()


def reference_main(args):
    """The oracle arm: the fp64 oracle as it stands on the host cores (all of them), each step
    a bounded sample of the same workload (see oracle_sample_text); one more step at one
    thread for the single-core figure. Rank 0 only; other ranks exit without work."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import torch
    wl = workload(args.workload)
    device = "cuda:0" if torch.cuda.is_available() else "cpu"
    import synth
    # weights drawn exactly as the GPU arm draws them (7B/13B shapes on the GPU)
    tw = synth.model_weights(wl, "target", device=device)
    dw = synth.model_weights(wl, "draft", device=device)
    cores = os.cpu_count()
    t_start = time.perf_counter()
    allc, one = oracle_runs(wl, tw, dw, args.oracle_layers,
                            [(cores, args.warmup, args.steps), (1, 0, 1)])
    wall = time.perf_counter() - t_start
    value = allc["tokens_per_step"] / allc["full_depth_step_s"]
    summ = lambda r: {"threads": r["threads"],
                      "sample_ms_per_step": round(r["sample_step_s"] * 1e3, 1),
                      "full_depth_ms_per_step_estimate": round(r["full_depth_step_s"] * 1e3, 1),
                      "tokens_per_s": round(r["tokens_per_step"] / r["full_depth_step_s"], 6)}
    out = {"metric": METRIC, "value": round(value, 6), "unit": "tokens/s", "n_gpus": 1,
           "steps": args.steps, "warmup": args.warmup,
           "ms_per_step": round(allc["sample_step_s"] * 1e3, 1),
           "ms_per_step_note": "measured: one sample step (the cut target); value uses the "
                               "full-depth estimate",
           "ms_per_step_full_depth_estimate": round(allc["full_depth_step_s"] * 1e3, 1),
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": "synthetic", "impl": "reference", "config": config_of(wl),
           "cpu_baseline": {"value": round(value, 6), "unit": "tokens/s", "kind": "oracle",
                            "cores": cores, "sample": oracle_sample_text(wl, args.oracle_layers),
                            "prefill_s": round(allc["prefill_s"], 1) if allc["prefill_s"] else None,
                            "all_cores": summ(allc), "one_thread": summ(one)},
           "e2e": {"value": round(value, 6), "unit": "tokens/s", "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0},
           "wall_s": round(wall, 1)}
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
    wbytes = streamed_weight_bytes_model(wl0.target)
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

    ints = lambda txt: [int(x) for x in txt.split(",") if x]
    for prefix in ints(args.sweep_prefix):
        t_dec = time_point(1, 1, prefix)
        for k in ints(args.sweep_k):
            for d in ints(args.sweep_d):
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
    if a.oracle_worker:
        oracle_worker(a)
    elif a.impl == "reference":
        reference_main(a)
    elif a.verify_sweep:
        verify_sweep(a)
    else:
        gpu_main(a)
