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
# DRAM bytes (read + write) per decode-GEMM launch: one ncu pass of dram__bytes_read.sum + dram__bytes_write.sum over
# the five decode GEMM shapes (QKV, O, gate/up, down, LM head) at 1024 and at 308 rows (the microbench's decode_gemms
# mode), weighted by a step's launches (32 layers x 4 + 1) and by the headline run's 443 steps at 1024 rows and 580
# at 308.  Algorithmic bytes of the same mix: 145.2 MB per launch.  Valid for the GEMM kernels as captured.
GEMM_DECODE_TRAFFIC = {"bytes_per_launch": 140.9e6, "algorithmic_bytes_per_launch": 145.2e6,
                       "source": "ncu dram__bytes_read.sum + dram__bytes_write.sum, decode GEMM shapes at 1024 / 308 rows"}


def load_peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        return {}


def aggregate_over_ranks(maxes, sums, world, device="cpu"):
    """Whole-job figures of one replica per rank: the max over ranks of each value in `maxes` (timed regions) and
    the sum over ranks of each value in `sums` (work done).  world <= 1 returns them unchanged."""
    maxes, sums = [float(x) for x in maxes], [float(x) for x in sums]
    if world <= 1:
        return maxes, sums
    import torch
    import torch.distributed as dist
    tm = torch.tensor(maxes, dtype=torch.float64, device=device)
    ts = torch.tensor(sums, dtype=torch.float64, device=device)
    dist.all_reduce(tm, op=dist.ReduceOp.MAX)
    dist.all_reduce(ts, op=dist.ReduceOp.SUM)
    return [float(x) for x in tm.tolist()], [float(x) for x in ts.tolist()]


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
def _median_time(fn, repeats=3):
    ts = []
    for _ in range(repeats):
        t0 = time.perf_counter()
        fn()
        ts.append(time.perf_counter() - t0)
    return statistics.median(ts)


class OracleUnitWork:
    """Unit work of the oracle timed on the host, extrapolated to a whole run.

    Timed: one decode step of a 1-layer model with the workload's widths at batch b = 4 and b = 16 and a
    CTX-position context (KV cache prefilled once), split into the layer (embedding, one transformer layer, final
    norm) and the head (LM head); and one reward-model chunk of 4 sequences of SCORE_P + SCORE_TAU positions
    through a 1-layer reward model.  Linear fits t(b) = a + c b give the decode cost of a run with S decode
    steps and G_dec tokens generated by them (G_dec = sum over steps of the live batch):
        T = L_gen (a_layer S + c_layer G_dec) + (a_head S + c_head G_dec) + L_rm c_score R,
    R = reward-model positions of the run (prompt once plus every scored partial or final response, as the
    library counts them; the oracle re-encodes the prompt per scored sequence, which is not counted, so T
    favours the oracle).  value = generated tokens / T."""
    CTX, SCORE_P, SCORE_TAU, BS = 512, 128, 64, (4, 16)

    def __init__(self, w: si.Workload, alpha: float, reward: str = "model"):
        from oracle.transformer import Decoder, Transformer
        self.w, self.alpha, self.reward = w, alpha, reward
        t0 = time.perf_counter()
        self.g = w.gen.replace(n_layers=1)
        self.gen = Transformer(self.g, si.random_weights(self.g, 100, 0))
        self.rm = None
        if reward == "model":
            self.r = w.rm.replace(n_layers=1)
            self.rm = Transformer(self.r, si.random_weights(self.r, 100, 1))
        self.ctx = min(self.CTX, w.gen.max_pos - 1)
        self.sp_len, self.tau = min(self.SCORE_P, w.rm.max_pos // 2), min(self.SCORE_TAU, w.rm.max_pos // 4)
        self.prompt = si.random_prompt(w.gen.vocab, self.ctx, 3)
        self.dec = Decoder(self.gen, max(self.BS), self.ctx + 1)
        self.dec.prefill(self.prompt, np.arange(max(self.BS)))
        self.setup_s = time.perf_counter() - t0
        try:
            import threadpoolctl
            self.cores = sum(p.get("num_threads", 0) for p in threadpoolctl.threadpool_info()
                             if p.get("user_api") == "blas") or os.cpu_count()
        except Exception:
            self.cores = os.cpu_count()
        self.units = None

    def measure(self, repeats: int = 3):
        from oracle.sr import score_sequences
        w, dec, ctx = self.w, self.dec, self.ctx
        t0 = time.perf_counter()
        layer, head = {}, {}
        for b in self.BS:
            toks = self.prompt[:b]
            hn = dec.step(np.arange(b), toks, ctx)
            layer[b] = _median_time(lambda: dec.step(np.arange(b), toks, ctx), repeats)
            head[b] = _median_time(lambda: self.gen.logits(hn), repeats)
        b0, b1 = self.BS
        c_l = (layer[b1] - layer[b0]) / (b1 - b0)
        c_h = (head[b1] - head[b0]) / (b1 - b0)
        u = {"a_layer": max(layer[b0] - c_l * b0, 0.0), "c_layer": c_l, "a_head": max(head[b0] - c_h * b0, 0.0),
             "c_head": c_h, "layer_s": layer, "head_s": head, "c_score": 0.0, "repeats": repeats}
        if self.rm is not None:
            sp = self.prompt[:self.sp_len]
            seqs = [list(si.random_prompt(w.gen.vocab, self.tau, 10 + i)) for i in range(4)]
            t = _median_time(lambda: score_sequences(self.rm, sp, seqs), repeats)
            u["score_chunk_s"] = t
            u["c_score"] = t / (4 * (self.sp_len + self.tau))
        u["measure_s"] = time.perf_counter() - t0
        self.units = u
        return u

    def extrapolate(self, S: float, G: float, A: float, R: float, what: str):
        """Oracle time of a run with S decode steps, G generated tokens (A of them sampled at admission from the
        prompt logits, no decode step) and R reward-model positions."""
        u = self.units or self.measure()
        Lg = self.w.gen.n_layers
        Lr = self.w.rm.n_layers if self.rm is not None else 0
        gd = G - A
        T = Lg * (u["a_layer"] * S + u["c_layer"] * gd) + (u["a_head"] * S + u["c_head"] * gd) + \
            Lr * u["c_score"] * R
        b0, b1 = self.BS
        sample = (f"oracle unit work on {self.w.name} widths ({self.reward} reward, alpha {self.alpha}): 1-layer decode "
                  f"step at b={b0} / b={b1}, context {self.ctx}: layer {u['layer_s'][b0]:.3f} / {u['layer_s'][b1]:.3f} s, "
                  f"LM head {u['head_s'][b0]:.3f} / {u['head_s'][b1]:.3f} s"
                  + (f"; 1-layer reward chunk of 4 x {self.sp_len}+{self.tau} positions {u['score_chunk_s']:.3f} s"
                     if self.rm is not None else "")
                  + f" (median of {u['repeats']}, {u['measure_s']:.0f} s of host work after {self.setup_s:.0f} s of "
                  f"model set-up). Extrapolated to {what}: "
                  f"T = {Lg} (a_l S + c_l G_dec) + (a_h S + c_h G_dec) + {Lr} c_s R with S = {S:.0f} decode steps, "
                  f"G_dec = {gd:.0f} tokens, R = {R:.0f} reward positions: T = {T:.0f} s for {G:.0f} tokens")
        return {"value": G / T, "unit": UNIT, "cores": self.cores, "kind": "oracle", "sample": sample,
                "oracle_s": T}


def expected_counts(w: si.Workload, P: int, alpha: float):
    """Decode steps, generated tokens, tokens sampled at admission and reward-model positions of one run on a
    P-token prompt when no candidate emits EOS (at this workload's EOS bias about 2 % of candidates stop early),
    under the pool reading of the library: 16-position pages, shared full prompt pages, one private tail page,
    a round at each fixed decision point or, memory-triggered, when the free pages cannot serve a step (k raised
    until they can), Best-of-N in pool-sized waves at alpha = 0 under a memory trigger.  Used by the CPU-only reference arm, which has no GPU run to count."""
    from oracle.pool import pool_pages, private_pages_full
    from oracle.select import cut_index
    n_pages = pool_pages(w.pool_bytes, si.kv_bytes_per_token(w.gen)) if w.pool_bytes else \
        P // 16 + w.N * private_pages_full(P, w.max_new)
    free = n_pages - P // 16
    per = private_pages_full(P, w.max_new)
    if alpha == 0.0:
        wave = min(w.N, free // per) if w.sched_kind == si.SCHED_POOL_FULL else w.N
        n_waves = -(-w.N // wave)
        return dict(S=n_waves * (w.max_new - 1), G=w.N * w.max_new, A=w.N, R=P + w.N * w.max_new)
    b, S, G, R = w.N, 0, w.N, P
    free -= b if P % 16 else 0
    for g in range(1, w.max_new):
        need = (P + g - 1) % 16 == 0
        trig = (g in w.taus) if w.sched_kind == si.SCHED_FIXED else (need and free < b)
        if trig:
            held = (P + g - 2) // 16 + 1 - P // 16
            R += b * g
            k = cut_index(alpha, b)
            while w.sched_kind != si.SCHED_FIXED and need and (b - k) > free + k * held and k < b - 1:
                k += 1
            free += k * held
            b -= k
        if need:
            free -= b
        S += 1
        G += b
    R += b * w.max_new
    return dict(S=S, G=G, A=w.N, R=R)


def run_reference(args, w):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    alpha = w.alpha if args.alpha is None else args.alpha
    unit = OracleUnitWork(w, alpha, args.reward)
    steps = []
    for k in range(args.warmup + args.steps):
        idx = k % max(1, w.n_prompts)
        P = len(w.prompt(idx))
        c = expected_counts(w, P, alpha)
        if args.reward != "model":
            c["R"] = 0
        unit.measure(repeats=1)                # every step times its own unit work
        s = unit.extrapolate(c["S"], c["G"], c["A"], c["R"], f"one response to prompt {idx} (P = {P}, "
                             f"counts of the run without EOS)")
        if k >= args.warmup:
            steps.append(s)
    tok = sum(s["value"] * s["oracle_s"] for s in steps)
    v = tok / sum(s["oracle_s"] for s in steps)
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * statistics.mean(s["oracle_s"] for s in steps),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": w.name, "alpha": alpha, "reward": args.reward, "sample": steps[0]["sample"]},
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
    ap.add_argument("--e2e-steps", type=int, default=2)
    ap.add_argument("--rm-cache-gb", type=float, default=64.0,
                    help="reward-model KV kept across rounds (sr_set_rm_cache), GB; 0 rescores every round in full")
    ap.add_argument("--bon-steps", type=int, default=1,
                    help="responses of the same path at alpha = 0 (Best-of-N in pool-sized waves) timed after the run")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--prof-period", type=int, default=8,
                    help="CUDA events around one launch in this many of each kernel class inside the timed region")
    ap.add_argument("--max-new", type=int, default=None,
                    help="shorter generations (a reduced case, e.g. for an ncu launch list of a whole response)")
    ap.add_argument("--pool-gb", type=float, default=None, help="KV pool size override, GB (with --max-new)")
    args = ap.parse_args()
    w = si.WORKLOADS[args.workload]
    if args.max_new is not None:
        w = w.replace(max_new=args.max_new)
    if args.pool_gb is not None:
        w = w.replace(pool_bytes=int(args.pool_gb * 1e9))
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
    sr.sr_set_rm_cache(ctx, int(args.rm_cache_gb * 1e9))
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
    (ms,), (gen_tokens, rm_tokens) = aggregate_over_ranks([ms], [gen_tokens, rm_tokens], world,
                                                         "cuda" if world > 1 else "cpu")
    value = gen_tokens / (ms / 1e3)

    # end to end through the public host API: prompt H2D and result D2H inside the timed region
    e2e = None
    if args.e2e_steps > 0:
        sr.sr_set_profiling(ctx, False)
        hp = [w.prompt(i) for i in range(n_prompts)]
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
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
        if world > 1:  # whole job: the slowest rank's wall time, every rank's tokens
            dist.barrier()
            (dt,), (e2e_tokens,) = aggregate_over_ranks([dt], [e2e_tokens], world, "cuda")
        e2e = {"value": e2e_tokens / dt, "unit": UNIT, "h2d_bytes_per_step": h2d // args.e2e_steps,
               "d2h_bytes_per_step": d2h // args.e2e_steps, "steps": args.e2e_steps,
               "ms_per_step": dt * 1e3 / args.e2e_steps}
    # Best-of-N baseline: the same library path with alpha = 0 (pool-sized waves), device buffers, own CUDA events
    bon = None
    if args.bon_steps > 0 and alpha > 0:
        sr.sr_set_profiling(ctx, False)
        torch.cuda.synchronize()
        b0, b1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        bst = []
        b0.record(stream)
        for k in range(args.bon_steps):
            p = prompts[(rank * (args.warmup + args.steps) + args.warmup + k) % n_prompts]
            bst.append(sr.sr_generate_dev(ctx, p, w.N, 0.0, w.sched_kind, w.taus, w.max_new, w.temperature,
                                          w.eos_bias, w.eos_id, args.warmup + k, out_tok, out_len, out_score, stream))
        b1.record(stream)
        torch.cuda.synchronize()
        bms = b0.elapsed_time(b1)
        btok = sum(s["gen_tokens"] for s in bst)
        bon = {"alpha": 0.0, "value": round(btok / (bms / 1e3), 1), "unit": UNIT,
               "wall_s_per_response": round(bms / args.bon_steps / 1e3, 3), "steps": args.bon_steps,
               "gen_tokens_per_response": btok // args.bon_steps, "waves": [s["waves"] for s in bst],
               "prompts": [int((rank * (args.warmup + args.steps) + args.warmup + k) % n_prompts)
                           for k in range(args.bon_steps)],
               "note": "Best-of-N baseline: the same libsr path with alpha = 0, run in KV-pool-sized waves "
                       "(same prompts as the first timed SR steps; CUDA events on the library's stream)"}
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
    if not dv["ms"]:  # --prof-period 0: no kernel was timed
        roof = None
    elif dom.startswith("gemm") or dom == "attn_prefill":
        achieved = dv["timed_flops"] / (dv["ms"] / 1e3) / 1e12
        tr = GEMM_DECODE_TRAFFIC if (dom == "gemm_decode" and w.name == "llama8b_n1024" and args.max_new is None
                                     and args.pool_gb is None) else None
        roof = {"bound": "tensor", "achieved": round(achieved, 1), "peak": tf_sus, "unit": "TFLOP/s",
                "frac": round(achieved / tf_sus, 4), "traffic": tr["bytes_per_launch"] if tr else None,
                "traffic_note": tr, "kernel": dom,
                "note": f"bf16 dense sustained peak ({src}); achieved = 2MNK per launch / CUDA-event launch time, "
                        f"over the {dv['timed']} launches timed (one in {args.prof_period} of each class)"}
    else:
        achieved = dv["timed_bytes"] / (dv["ms"] / 1e3) / 1e9
        roof = {"bound": "hbm", "achieved": round(achieved, 1), "peak": hbm, "unit": "GB/s",
                "frac": round(achieved / hbm, 4), "traffic": None, "kernel": dom, "note": f"HBM copy peak ({src})"}
    ad = kern["attn_decode"]
    if ad["ms"] and roof is not None:
        gbs = ad["timed_bytes"] / (ad["ms"] / 1e3) / 1e9
        roof["attn_decode"] = {"bound": "hbm", "achieved": round(gbs, 1), "peak": hbm, "unit": "GB/s",
                               "frac": round(gbs / hbm, 4), "frac_of_8tbs_nominal": round(gbs / 8000.0, 4)}
    clocks = clk.summary()
    s0 = stats[0]
    line = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms / args.steps, 1), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f16", "data": "synthetic",
        "config": {"workload": w.name, "model": "Llama-3-8B-shaped generator + reward model (random-init bf16)",
                   "N": w.N, "alpha": alpha, "reward": args.reward, "schedule": "memory-triggered" if w.sched_kind else f"tau={w.taus}",
                   "kv_pool_bytes": w.pool_bytes, "rm_cache_bytes": int(args.rm_cache_gb * 1e9), "max_new": w.max_new, "temperature": w.temperature,
                   "eos_bias": w.eos_bias, "global_batch": w.N * world, "seq_len": f"P~U[{w.prompt_len_min},"
                   f"{w.prompt_len}] + {w.max_new}", "parallelism": f"replicas x{world}",
                   "l2": "inputs larger than L2 (16 GB of weights per model read every step)",
                   "precision": "bf16 weights converted once to fp16 at sr_init; fp16 tensor-core operands and KV "
                                "cache, fp32 accumulation, softmax, norms and residual stream",
                   "prompts_timed": [int((rank * (args.warmup + args.steps) + args.warmup + k) % n_prompts)
                                     for k in range(args.steps)]},
        "wall_s_per_response": round(ms / args.steps / 1e3, 3),
        "rm_tokens_per_s": round(rm_tokens / (ms / 1e3), 1),
        "rm_tokens_cached_per_response": sum(s["rm_tokens_cached"] for s in stats) // args.steps,
        "rounds": [s["rounds"] for s in stats], "b_per_round": [s["b_per_round"] for s in stats],
        "step_per_round": [s["step_per_round"] for s in stats],
        "roofline": roof, "kernels": summary,
        "gpu_launches": int(sum(v["launches"] for v in kern.values())),
        "clocks": clocks, "e2e": e2e,
    }
    if bon is not None:
        line["best_of_n"] = bon
        line["sr_speedup_vs_best_of_n"] = round(bon["wall_s_per_response"] / (ms / args.steps / 1e3), 3)
    if world == 1 and not args.no_cpu_baseline:
        S = sum(s["decode_steps"] for s in stats)
        A = w.N * len(stats)
        line["cpu_baseline"] = OracleUnitWork(w, alpha, args.reward).extrapolate(
            S, gen_tokens, A, rm_tokens, f"the {args.steps} timed responses (their own decode-step, token and "
            f"reward-position counts)")
    print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
