"""Benchmark: Speculative Rejection on the Llama-3-8B-shaped workload, N = 1024 candidates.

One step = one full sr_generate (Algorithm 1: prompt prefill, batched decode of 1024 candidates,
memory-triggered rejection rounds, partial / final reward scoring, selection) for one prompt of
the workload's 8 synthetic prompts.  Inputs (weights, prompts) are resident in HBM before the
timed region; the 16 GB of weights per model keep every step's working set far above the 129 MB
L2, so no explicit flush is needed.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--workload NAME]

Under torchrun each rank runs an independent replica on its own prompts (the method does not
shard: one prompt is one GPU's work); rank 0 prints one JSON line.  --impl reference times the
CPU oracle (oracle/) on a bounded sample of the same workload on the host cores.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np

import sr_inputs as si

METRIC = "Best-of-N wall time & generated tokens/s at 8B, N=1024; HBM roofline %"
UNIT = "generated tokens/s"
KC = ("gemm_decode", "gemm_score", "gemm_prompt", "attn_decode", "attn_prefill", "sample", "elementwise", "control")


def load_peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        return {}


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


class ClockSampler:
    """nvidia-smi clock / throttle samples while the timed region runs."""

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
             "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
             "clocks_event_reasons.sw_power_cap")
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        rows = []
        try:
            for line in open(self.path):
                f = [x.strip() for x in line.split(",")]
                if len(f) >= 9 and f[1].isdigit():
                    rows.append(f)
        except Exception:
            pass
        finally:
            if self.path and os.path.exists(self.path):
                os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        sm = [int(r[1]) for r in rows]
        mx = int(rows[0][2])
        loaded = [r for r in rows if float(r[3]) > 200.0] or rows
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(int(r[1]) for r in loaded), "sm_max_mhz": mx, "reasons": reasons,
                "samples": len(rows), "sm_mhz_min": min(sm)}


# ------------------------------------------------------------------------------------------------
# CPU oracle sample (cpu_baseline and --impl reference)
# ------------------------------------------------------------------------------------------------
class OracleSample:
    """The oracle's Algorithm 1 on a bounded sample of the workload: the same widths, vocabulary and heads, 1 of
    the 32 layers, 2 candidates, a 64-token prompt prefix, 4 new tokens, one decision point at 2.  Its tokens/s
    is scaled to the full models by the ratio of matmul parameters touched per generated token (generator +
    reward model), i.e. assuming cost linear in layers.  Models are built once; each run is timed."""
    L, N, MAX_NEW, P = 1, 2, 4, 64

    def __init__(self, w: si.Workload, alpha=None, reward: str = "model"):
        from oracle.transformer import Transformer
        self.w = w
        self.alpha = w.alpha if alpha is None else alpha
        self.reward = reward
        self.g = w.gen.replace(n_layers=self.L)
        self.r = w.rm.replace(n_layers=self.L)
        self.gen = Transformer(self.g, si.random_weights(self.g, 100, 0))
        self.rm = Transformer(self.r, si.random_weights(self.r, 100, 1))

        def per_tok(m):
            layer = m.qkv_dim * m.d_model + m.d_model * m.n_heads * m.head_dim + \
                (3 if m.gated else 2) * m.ffn_dim * m.d_model
            return m.n_layers * layer + (m.vocab * m.d_model if m.has_lm_head else m.d_model)
        with_rm = reward == "model"  # the self-likelihood reward runs no reward model
        self.scale = (per_tok(w.gen) + with_rm * per_tok(w.rm)) / (per_tok(self.g) + with_rm * per_tok(self.r))
        try:
            import threadpoolctl
            self.cores = sum(p.get("num_threads", 0) for p in threadpoolctl.threadpool_info()
                             if p.get("user_api") == "blas") or os.cpu_count()
        except Exception:
            self.cores = os.cpu_count()

    def run(self, prompt_index: int = 0):
        from oracle.sr import SpeculativeRejection
        w = self.w
        prompt = w.prompt(prompt_index)[:self.P]
        t0 = time.perf_counter()
        res = SpeculativeRejection(self.gen, self.rm, prompt, self.N, self.alpha, si.SCHED_FIXED, (2,), self.MAX_NEW,
                                   w.temperature, w.eos_bias, w.eos_id, 0, reward=self.reward).run()
        dt = time.perf_counter() - t0
        return {"value": res.gen_tokens / dt / self.scale, "unit": UNIT, "cores": self.cores, "kind": "oracle",
                "sample": (f"oracle Algorithm 1 ({self.reward} reward, alpha {self.alpha}) on {w.name} widths with "
                           f"{self.L}/{w.gen.n_layers} layers, "
                           f"N={self.N}, P={len(prompt)}, {self.MAX_NEW} new tokens, one round at 2: "
                           f"{res.gen_tokens} tokens in {dt:.1f} s on the host, scaled by 1/{self.scale:.1f} "
                           f"(matmul parameters per token, full / sample)")}


def run_reference(args, w):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    smp = OracleSample(w, args.alpha, args.reward)
    steps = []
    for k in range(args.warmup + args.steps):
        s = smp.run(k % max(1, w.n_prompts))
        if k >= args.warmup:
            steps.append(s)
    v = statistics.mean(s["value"] for s in steps)
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": None, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": w.name, "sample": steps[0]["sample"]},
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": steps[0]["cores"], "kind": "oracle",
                             "sample": steps[0]["sample"]},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------------------------------------
# our arm
# ------------------------------------------------------------------------------------------------
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="llama8b_n1024", choices=sorted(si.WORKLOADS))
    ap.add_argument("--alpha", type=float, default=None, help="override the rejection rate (0 = Best-of-N)")
    ap.add_argument("--reward", default="model", choices=["model", "logprob"],
                    help="reward model, or the generator's mean log-probability (Section 5.3)")
    ap.add_argument("--e2e-steps", type=int, default=1)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--prof-period", type=int, default=8,
                    help="CUDA events around one launch in this many of each kernel class inside the timed region")
    args = ap.parse_args()
    w = si.WORKLOADS[args.workload]
    if args.impl == "reference":
        return run_reference(args, w)

    import torch
    import torch.distributed as dist
    from paper_2410_20290_gb300 import binding as sr

    rank, world, local = dist_env()
    if world > 1:
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    torch.cuda.set_device(local)
    alpha = w.alpha if args.alpha is None else args.alpha

    # weights: random-init bf16, drawn on the device (inputs, resident before timing)
    if w.gen.dtype == si.DT_BF16 and si.n_params(w.gen) > 50_000_000:
        gblob = si.device_weight_blob(w.gen, w.weight_seed, 0)
        rblob = si.device_weight_blob(w.rm, w.weight_seed, 1)
    else:
        gblob = torch.from_numpy(si.pack_blob(w.gen, si.random_weights(w.gen, w.weight_seed, 0))).cuda()
        rblob = torch.from_numpy(si.pack_blob(w.rm, si.random_weights(w.rm, w.weight_seed, 1))).cuda()
    ctx = sr.sr_init(w.gen, gblob, w.rm, rblob, w.pool_bytes, 16, local)
    del gblob, rblob
    torch.cuda.empty_cache()
    stream = torch.cuda.Stream()
    sr.sr_set_stream(ctx, stream)
    sr.sr_set_reward(ctx, sr.SR_REWARD_LOGPROB if args.reward == "logprob" else sr.SR_REWARD_MODEL)
    n_prompts = max(1, w.n_prompts)
    prompts = [torch.from_numpy(w.prompt(i)).cuda() for i in range(n_prompts)]
    out_tok = torch.zeros(w.max_new, dtype=torch.int32, device="cuda")
    out_len = torch.zeros(1, dtype=torch.int32, device="cuda")
    out_score = torch.zeros(1, dtype=torch.float32, device="cuda")

    def step(k, profile):
        p = prompts[(rank * (args.warmup + args.steps) + k) % n_prompts]
        sr.sr_set_profiling(ctx, profile)
        return sr.sr_generate_dev(ctx, p, w.N, alpha, w.sched_kind, w.taus, w.max_new, w.temperature, w.eos_bias,
                                  w.eos_id, k, out_tok, out_len, out_score, stream)

    for k in range(args.warmup):
        step(k, False)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    stats = []
    with ClockSampler(local) as clk:
        ev0.record(stream)
        for k in range(args.steps):
            stats.append(step(args.warmup + k, args.prof_period))
        ev1.record(stream)
        torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    ms = ev0.elapsed_time(ev1)
    gen_tokens = sum(s["gen_tokens"] for s in stats)
    rm_tokens = sum(s["rm_tokens"] for s in stats)
    t = torch.tensor([ms, gen_tokens, rm_tokens], dtype=torch.float64, device="cuda")
    if world > 1:
        tmax = t.clone()
        dist.all_reduce(tmax[:1], op=dist.ReduceOp.MAX)
        tsum = t.clone()
        dist.all_reduce(tsum, op=dist.ReduceOp.SUM)
        ms, gen_tokens, rm_tokens = float(tmax[0]), float(tsum[1]), float(tsum[2])
    value = gen_tokens / (ms / 1e3)

    # end to end through the public host API: prompt H2D and result D2H inside the timed region
    e2e = None
    if args.e2e_steps > 0:
        sr.sr_set_profiling(ctx, False)
        hp = [w.prompt(i) for i in range(n_prompts)]
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        e2e_tokens, h2d, d2h = 0, 0, 0
        for k in range(args.e2e_steps):
            p = hp[(args.warmup + args.steps + k) % n_prompts]
            toks, score, st = sr.sr_generate(ctx, p, w.N, alpha, w.sched_kind, w.taus, w.max_new, w.temperature,
                                             w.eos_bias, w.eos_id, 1000 + k)
            e2e_tokens += st["gen_tokens"]
            h2d += p.nbytes
            d2h += toks.nbytes + 8
        dt = time.perf_counter() - t0
        e2e = {"value": e2e_tokens / dt, "unit": UNIT, "h2d_bytes_per_step": h2d // args.e2e_steps,
               "d2h_bytes_per_step": d2h // args.e2e_steps, "steps": args.e2e_steps,
               "ms_per_step": dt * 1e3 / args.e2e_steps}
    sr.sr_destroy(ctx)
    if rank != 0:
        return

    peaks = load_peaks()
    hbm = peaks.get("hbm_gbs", 6800.0)
    tf_sus = peaks.get("bf16_tflops_sustained", 1700.0)
    src = "of measured" if peaks else "of fallback"
    # per kernel class: every launch is counted; one in --prof-period is timed with CUDA events, and the
    # class's time is estimated as (timed time) x launches / timed launches
    kern = {c: dict(ms=0.0, launches=0, flops=0.0, bytes=0.0, timed=0, timed_flops=0.0, timed_bytes=0.0) for c in KC}
    for s in stats:
        for c in KC:
            for f in kern[c]:
                kern[c][f] += s["kernels"][c][f]
    for v in kern.values():
        v["est_ms"] = v["ms"] * v["launches"] / v["timed"] if v["timed"] else 0.0
    total_k = sum(v["est_ms"] for v in kern.values()) or 1.0
    summary = {}
    for c, v in kern.items():
        if v["launches"] == 0:
            continue
        sec = v["ms"] / 1e3
        e = {"ms": round(v["est_ms"], 1), "share": round(v["est_ms"] / total_k, 4), "launches": v["launches"],
             "timed": v["timed"]}
        if v["timed_flops"] and sec:
            e["tflops"] = round(v["timed_flops"] / sec / 1e12, 1)
        if v["timed_bytes"] and sec:
            e["gbs"] = round(v["timed_bytes"] / sec / 1e9, 1)
        summary[c] = e
    dom = max(kern, key=lambda c: kern[c]["est_ms"])
    dv = kern[dom]
    if dom.startswith("gemm") or dom == "attn_prefill":
        achieved = dv["timed_flops"] / (dv["ms"] / 1e3) / 1e12
        roof = {"bound": "tensor", "achieved": round(achieved, 1), "peak": tf_sus, "unit": "TFLOP/s",
                "frac": round(achieved / tf_sus, 4), "traffic": None, "kernel": dom,
                "note": f"bf16 dense sustained peak ({src}); achieved = 2MNK per launch / CUDA-event launch time, "
                        f"over the {dv['timed']} launches timed (one in {args.prof_period} of each class)"}
    else:
        achieved = dv["timed_bytes"] / (dv["ms"] / 1e3) / 1e9
        roof = {"bound": "hbm", "achieved": round(achieved, 1), "peak": hbm, "unit": "GB/s",
                "frac": round(achieved / hbm, 4), "traffic": None, "kernel": dom, "note": f"HBM copy peak ({src})"}
    ad = kern["attn_decode"]
    if ad["ms"]:
        gbs = ad["timed_bytes"] / (ad["ms"] / 1e3) / 1e9
        roof["attn_decode"] = {"bound": "hbm", "achieved": round(gbs, 1), "peak": hbm, "unit": "GB/s",
                               "frac": round(gbs / hbm, 4), "frac_of_8tbs_nominal": round(gbs / 8000.0, 4)}
    clocks = clk.summary()
    s0 = stats[0]
    line = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms / args.steps, 1), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": w.name, "model": "Llama-3-8B-shaped generator + reward model (random-init bf16)",
                   "N": w.N, "alpha": alpha, "reward": args.reward, "schedule": "memory-triggered" if w.sched_kind else f"tau={w.taus}",
                   "kv_pool_bytes": w.pool_bytes, "max_new": w.max_new, "temperature": w.temperature,
                   "eos_bias": w.eos_bias, "global_batch": w.N * world, "seq_len": f"P~U[{w.prompt_len_min},"
                   f"{w.prompt_len}] + {w.max_new}", "parallelism": f"replicas x{world}",
                   "l2": "inputs larger than L2 (16 GB of weights per model read every step)",
                   "prompts_timed": [int((rank * (args.warmup + args.steps) + args.warmup + k) % n_prompts)
                                     for k in range(args.steps)]},
        "wall_s_per_response": round(ms / args.steps / 1e3, 3),
        "rm_tokens_per_s": round(rm_tokens / (ms / 1e3), 1),
        "rounds": [s["rounds"] for s in stats], "b_per_round": [s["b_per_round"] for s in stats],
        "step_per_round": [s["step_per_round"] for s in stats],
        "roofline": roof, "kernels": summary,
        "gpu_launches": int(sum(v["launches"] for v in kern.values())),
        "clocks": clocks, "e2e": e2e,
    }
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = OracleSample(w, alpha, args.reward).run(0)
    print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
