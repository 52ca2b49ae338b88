#!/usr/bin/env python3
"""Benchmark: time-to-first-token of restoration-overlapped prefill on GB300.

One step = one TTFT: mzc_restore_async -> mzc_recompute_tail -> mzc_prefill
(prompt) -> first-token logits in host memory, over a context whose evicted
part was put back at rest (evicted) before the step, outside the timed region
(the paper's TTFT includes restoration but not eviction, Sec. 6.1).

Workloads (synthetic stand-ins for the paper's models, see synth/workloads.py):
  1b_recompute (default)  16L d2048, 8192-token context, tail [4096, 8192)
                          dropped and recomputed, 128-token prompt
  tiny                    2L d256, 512-token context, tail 256 dropped, 32-token prompt
  3b_scattered_copy       28L d3072, 32768-token context, 30% of blocks swapped to
                          pinned host and copied back while the prompt (256) runs
  3b_mixed                28L, last 8 layers' weights streamed, tail >= 16384 dropped,
                          20% of the rest copied, 512-token prompt
  3b_sweep                28L, evicted fraction {0,10,25,50,75,100}% x {copy, recompute,
                          hybrid}, 128-token prompt (one JSON line per point, to stderr)

value: device TTFT (CUDA events: start of the restore copies, or of the prefill when
nothing is copied, to the logits landing in host memory), median over the timed steps.
e2e: the same TTFT on the host clock through the C ABI with host buffers.
--impl reference: the CPU oracle (the repo's plain fp32 restatement) timed on a
bounded sample of the same workload, scaled to the whole step.
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

METRIC = "TTFT ms vs evicted fraction (1 GB300); recompute tok/s; % BF16 tensor peak"


def _traffic(kernel_class, workload):
    """Per-launch DRAM bytes from the committed ncu capture, or None when the
    capture was of another workload or the kernel's source changed since the
    counters were taken."""
    import hashlib
    try:
        with open(os.path.join(ROOT, "profiles", "ncu_traffic.json")) as f:
            t = json.load(f)[kernel_class]
        if t.get("workload") != workload:
            return None
        src = open(os.path.join(ROOT, t["source"]), "rb").read()
        if hashlib.sha256(src).hexdigest()[:16] != t["source_sha"]:
            return None
        return t["bytes_per_launch"]
    except Exception:
        return None


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return p, "measured"
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


class Clocks:
    """nvidia-smi sampling during the timed region."""

    def __init__(self, index: int):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.p = subprocess.Popen(["nvidia-smi", f"--id={index}", f"--query-gpu={q}",
                                       "--format=csv,noheader,nounits", "-lms", "200"],
                                      stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.p = None

    def stop(self):
        if self.p is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.p.terminate()
        self.p.wait()
        self.f.flush()
        self.f.seek(0)
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.f.read().splitlines():
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = float(parts[2])
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        os.unlink(self.f.name)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm)}


# ---- workloads -----------------------------------------------------------------

def _workload(name):
    from synth import workloads as W
    sc = dict(W.SCENARIOS["1b_recompute" if name == "1b_recompute" else name])
    return sc


def _describe(name, sc):
    m = sc["model"]
    base = (f"{m['n_layers']}L d{m['d_model']} {m['n_q_heads']}/{m['n_kv_heads']}x{m['head_dim']} "
            f"F{m['ffn_dim']} V{m['vocab']} {'fp16' if m['kv_dtype'] == 1 else 'bf16'} KV; "
            f"context {sc['context']}")
    if name in ("1b_recompute", "tiny"):
        return f"{name}: {base}, tail [{sc['context'] - sc['evict_tail']},{sc['context']}) dropped and recomputed, {sc['prompt']}-token prompt"
    if name == "3b_scattered_copy":
        return f"{name}: {base}, {int(sc['scatter_frac'] * 100)}% of KV blocks swapped to pinned host and copied back, {sc['prompt']}-token prompt"
    if name == "3b_mixed":
        return (f"{name}: {base}, weights of layers {sc['weights_evicted'][0]}-{sc['weights_evicted'][1] - 1} streamed, "
                f"tail >= {sc['drop_from']} recomputed, {int(sc['scatter_frac'] * 100)}% of the rest copied, {sc['prompt']}-token prompt")
    return f"{name}: {base}"


class Runner:
    """Owns one ctx on one GPU and knows how to put the evicted state at rest
    (untimed) and run one timed restore + prefill."""

    def __init__(self, name, sc, device, codec=0):
        import synth
        import paper_2609_01338_gb300 as m
        self.m, self.name, self.sc = m, name, sc
        sh = sc["model"]
        self.shape = sh
        t = time.time()
        self.w = synth.model_weights(sh)
        self.t_gen = time.time() - t
        self.ctx_tokens = synth.tokens(synth.SEED_CONTEXT, 0, sc["context"], sh["vocab"])
        self.prompt = synth.tokens(synth.SEED_PROMPT, 0, sc["prompt"], sh["vocab"])
        max_rows = min(sh["max_ctx"], 16384 + 1024)
        t = time.time()
        self.c = m.mzc_create(sh, self.w, max_rows=max_rows, device=device, swap_codec=codec)
        self.t_create = time.time() - t
        t = time.time()
        m.mzc_prefill(self.c, self.ctx_tokens)  # long contexts run in causal chunks
        self.t_ctx = time.time() - t
        self.logits = np.empty(sh["vocab"], np.float32)
        self.N = sc["context"]
        L = sh["n_layers"]
        self.nblk = -(-self.N // 16)
        self.rec = None
        if name == "3b_scattered_copy" or name == "3b_mixed":
            import synth as S
            if name == "3b_scattered_copy":
                pairs = L * self.nblk
                k = int(round(sc["scatter_frac"] * pairs))
                sel = S.permutation(S.SEED_EVICT, 0, pairs)[:k]
                self.scatter = (sel // self.nblk, sel % self.nblk)
            else:
                eligible = sc["drop_from"] // 16
                pairs = L * eligible
                k = int(round(sc["scatter_frac"] * pairs))
                sel = S.permutation(S.SEED_EVICT, 1, pairs)[:k]
                self.scatter = (sel // eligible, sel % eligible)

    def evict(self, policy=None, frac=None):
        m, L, N = self.m, self.shape["n_layers"], self.N
        self.rec = None
        if self.name in ("1b_recompute", "tiny"):
            p = N - self.sc["evict_tail"]
            m.mzc_evict(self.c, 0, L, p, N, m.MZC_DROP)
            self.rec = (p, N - p)
        elif self.name == "3b_scattered_copy":
            m.mzc_evict_blocks(self.c, self.scatter[0], self.scatter[1])
        elif self.name == "3b_mixed":
            a, b = self.sc["weights_evicted"]
            m.mzc_evict_weights(self.c, a, b)
            m.mzc_evict_blocks(self.c, self.scatter[0], self.scatter[1])
            p = self.sc["drop_from"]
            m.mzc_evict(self.c, 0, L, p, N, m.MZC_DROP)
            self.rec = (p, N - p)
        elif self.name == "3b_sweep":
            n_ev = int(np.ceil(frac * self.nblk)) * 16
            p = max(0, N - n_ev)
            if n_ev == 0:
                return
            if policy == "copy":
                m.mzc_evict(self.c, 0, L, p, N, m.MZC_COPY)
            elif policy == "recompute":
                m.mzc_evict(self.c, 0, L, p, N, m.MZC_DROP)
                self.rec = (p, N - p)
            else:
                s = m.mzc_plan_split_ctx(self.c, p, self.sc["prompt"])
                if s > p:
                    m.mzc_evict(self.c, 0, L, p, s, m.MZC_DROP)
                    self.rec = (p, s - p)
                if s < N:
                    m.mzc_evict(self.c, 0, L, s, N, m.MZC_COPY)

    def step(self):
        m = self.m
        t0 = time.perf_counter()
        m.mzc_restore_async(self.c)
        if self.rec:
            m.mzc_recompute_tail(self.c, *self.rec)
        m.mzc_prefill(self.c, self.prompt, self.logits)
        t1 = time.perf_counter()
        times = m.mzc_last_times(self.c)
        st = m.mzc_stats(self.c)
        m.mzc_truncate(self.c, self.N)
        return float(times[3]), (t1 - t0) * 1e3, st, times

    def close(self):
        self.m.mzc_destroy(self.c)


_ORACLE_WEIGHTS = {}


def _cpu_sample(sc, n_rows_sample):
    """Times the oracle on a bounded sample of the step's rows (all layers,
    over a zero KV state of the workload's shape) and scales it to the step:
    ms = t(sample rows) * rows / sample + t(LM head on one row)."""
    import oracle
    import synth
    sh = sc["model"]
    N, P = sc["context"], sc["prompt"]
    if "evict_tail" in sc:
        rec = sc["evict_tail"]
    elif "drop_from" in sc:
        rec = N - sc["drop_from"]
    else:
        rec = 0
    rows_pos = np.concatenate([np.arange(N - rec, N), np.arange(N, N + P)]).astype(np.int64)
    total = rows_pos.size
    idx = np.unique(np.linspace(0, total - 1, min(n_rows_sample, total)).astype(int))
    key = tuple(sorted((k, v) for k, v in sh.items()))
    if key not in _ORACLE_WEIGHTS:
        _ORACLE_WEIGHTS.clear()
        _ORACLE_WEIGHTS[key] = synth.model_weights(sh)
    w = _ORACLE_WEIGHTS[key]
    ctx_len = N + P
    kv = oracle.KVState.__new__(oracle.KVState)
    dims = (sh["n_layers"], ctx_len, sh["n_kv_heads"], sh["head_dim"])
    kv.k = np.zeros(dims, np.float32)
    kv.v = np.zeros(dims, np.float32)
    kv.max_ctx = ctx_len
    toks = synth.tokens(synth.SEED_PROMPT, 9, idx.size, sh["vocab"])
    t = time.perf_counter()
    oracle.forward(sh, w, kv, toks, rows_pos[idx], logits=False)
    t_rows = time.perf_counter() - t
    x = np.ones((1, sh["d_model"]), np.float32)
    t = time.perf_counter()
    h = oracle.rmsnorm(x, w["final_norm"], sh["rms_eps"])
    oracle.linear(h, w["lm_head"])
    t_lm = time.perf_counter() - t
    ms = (t_rows * total / idx.size + t_lm) * 1e3
    sample = (f"{idx.size} of {total} rows (evenly spaced over the recomputed tail and the prompt) "
              f"through all {sh['n_layers']} layers over a zero KV state of {ctx_len} positions, "
              f"scaled x{total / idx.size:.1f}, plus one LM-head row; {t_rows + t_lm:.1f} s of wall time")
    return ms, sample, oracle.num_threads()


def run_reference(args, name, sc, rank):
    if rank != 0:
        return
    import oracle
    oracle.build()
    vals = []
    sample = ""
    for i in range(args.warmup + args.steps):
        ms, sample, cores = _cpu_sample(sc, 8)
        if i >= args.warmup:
            vals.append(ms)
    v = statistics.median(vals)
    line = {"impl": "reference", "metric": METRIC, "value": round(v, 3), "unit": "ms",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(statistics.mean(vals), 3), "higher_is_better": False,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": _describe(name, sc)},
            "cpu_baseline": {"value": round(v, 3), "unit": "ms", "cores": cores,
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": round(v, 3), "unit": "ms", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="mzc", choices=["mzc", "reference"])
    ap.add_argument("--workload", default="1b_recompute",
                    choices=["1b_recompute", "tiny", "3b_scattered_copy", "3b_mixed", "3b_sweep",
                             "3b_order", "1b_decode", "3b_decode"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-kernel-timing", action="store_true")
    ap.add_argument("--fractions", default=None, help="comma list overriding the sweep's fractions")
    ap.add_argument("--policies", default=None, help="comma list overriding the sweep's policies")
    ap.add_argument("--codec", default="none", choices=["none", "q8"],
                    help="swap codec of the pinned store: none, or 8-bit groups (q8)")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "mzc":
        args.warmup = 3

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    name = args.workload
    sc = _workload(name)
    if args.fractions:
        sc["fractions"] = tuple(float(x) for x in args.fractions.split(","))
    if args.policies:
        sc["policies"] = tuple(args.policies.split(","))

    if args.impl == "reference":
        run_reference(args, name, sc, rank)
        return

    import torch
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU")
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")

    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_01338_gb300 as m

    r = Runner(name, sc, local, codec=1 if args.codec == "q8" else 0)
    if name == "3b_sweep":
        r.profile = m.mzc_profile_measure(r.c)
        run_sweep(r, args, rank)
        r.close()
        return
    if name == "3b_order":
        run_order(r, args, rank)
        r.close()
        return
    if name.endswith("_decode"):
        run_decode(r, args, rank)
        r.close()
        return
    # warm-up; the last warm-up step times every kernel class to find the
    # dominant one, and only that class is bracketed with events in the timed
    # steps (fewer events, less perturbation of the TTFT)
    warm_ks = {}
    for i in range(args.warmup):
        if i == args.warmup - 1:
            m.mzc_set_kernel_timing(r.c, -1)
        r.evict()
        r.step()
    warm_ks = {nm: m.mzc_kernel_stats(r.c, i) for i, nm in enumerate(m.KERNEL_CLASS_NAMES)}
    dom = max(warm_ks, key=lambda nm: warm_ks[nm].ms)
    m.mzc_set_kernel_timing(r.c, 0)
    if not args.no_kernel_timing:
        m.mzc_set_kernel_timing(r.c, 1 << m.KERNEL_CLASS_NAMES.index(dom))
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    clk = Clocks(local)
    dev, host, stats = [], [], None
    t_all = time.perf_counter()
    for _ in range(args.steps):
        r.evict()
        d, h, st, times = r.step()
        dev.append(d)
        host.append(h)
        stats = st
    torch.cuda.synchronize()
    wall = time.perf_counter() - t_all
    clocks = clk.stop()
    if dist:
        dist.barrier()
    ks = {nm: m.mzc_kernel_stats(r.c, i) for i, nm in enumerate(m.KERNEL_CLASS_NAMES)}
    m.mzc_set_kernel_timing(r.c, 0)

    v, e2e = max_over_ranks([statistics.median(dev), statistics.median(host)], dist, "cuda")

    peaks, src = _peaks()
    launches = sum(k.launches for k in ks.values())
    # the dominant kernel class (from the warm-up), timed live in the timed steps
    roof = None
    if not args.no_kernel_timing:
        k = ks[dom]
        per = k.launches if k.launches else 1
        # the bound follows the launches' arithmetic intensity: below the ridge
        # (sustained FLOP/s over HBM bytes/s) a contraction streams its operands
        ridge = peaks["bf16_tflops_sustained"] * 1e12 / (peaks["hbm_gbs"] * 1e9)
        tensor_bound = dom in ("gemm", "attention") and (k.bytes <= 0 or k.flops / k.bytes >= ridge)
        if tensor_bound:
            ach = k.flops / (k.ms * 1e-3) / 1e12
            peak = peaks["bf16_tflops_sustained"]
            roof = {"kernel": dom, "bound": "tensor", "achieved": round(ach, 2), "peak": peak,
                    "unit": "TFLOP/s", "frac": round(ach / peak, 4), "traffic": _traffic(dom, name),
                    "peak_source": f"{src} bf16 sustained (fp16 operands: nominal fp16/bf16 ratio 1.0)",
                    "avg_launch_ms": round(k.ms / per, 4), "flops_per_launch": k.flops / per}
        else:
            ach = k.bytes / (k.ms * 1e-3) / 1e9
            peak = peaks["hbm_gbs"]
            roof = {"kernel": dom, "bound": "hbm", "achieved": round(ach, 1), "peak": peak,
                    "unit": "GB/s", "frac": round(ach / peak, 4), "traffic": _traffic(dom, name),
                    "peak_source": f"{src} HBM copy", "avg_launch_ms": round(k.ms / per, 4),
                    "bytes_per_launch": k.bytes / per}
    rows = stats.rows_last
    rec_rows = stats.recompute_rows_last
    g = warm_ks["gemm"]
    gemm_tfs = g.flops / (g.ms * 1e-3) / 1e12 if g.ms > 0 else None
    a = warm_ks["attention"]
    attn_tfs = a.flops / (a.ms * 1e-3) / 1e12 if a.ms > 0 else None
    h2d = int(rows * 8 + sc["model"]["n_layers"] * (-(-sc["model"]["max_ctx"] // 16)) * 4
              + sc["prompt"] * 4 + stats.bytes_h2d_last)
    d2h = int(sc["model"]["vocab"] * 4)
    line = {
        "metric": METRIC, "value": round(v, 3), "unit": "ms", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(statistics.mean(dev), 3), "higher_is_better": False,
        "scaling": "weak", "vs_baseline": None, "dtype": "f16",
        "data": "synthetic (seeded N(0,0.02) bf16 weights, uniform token ids)",
        "config": {"workload": _describe(name, sc), "swap_codec": args.codec,
                   "l2": "inputs larger than L2 (weights + KV >> 129 MB)",
                   "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
                   "timed": "restore + recompute + prompt prefill + logits D2H per step; eviction between steps untimed"},
        "recompute_tok_s": round(rec_rows / (v * 1e-3), 1) if rec_rows else None,
        "rows_per_step": rows,
        "gemm_tflops": round(gemm_tfs, 1) if gemm_tfs else None,
        "attention_tflops": round(attn_tfs, 1) if attn_tfs else None,
        "tensor_peak_frac_gemm": round(gemm_tfs / peaks["bf16_tflops_sustained"], 4) if gemm_tfs else None,
        "kernel_ms_per_step": {n: round(k.ms, 3) for n, k in warm_ks.items()},
        "kernel_ms_source": "last warm-up step, every class timed",
        "roofline": roof,
        "e2e": {"value": round(e2e, 3), "unit": "ms", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        "gpu_launches": int(launches),
        "clocks": clocks,
        "wall_s_timed": round(wall, 2),
        "setup_s": {"weights": round(r.t_gen, 1), "create": round(r.t_create, 1),
                    "context_prefill": round(r.t_ctx, 2)},
    }
    r.close()
    del r
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        ms, sample, cores = _cpu_sample(sc, 32)
        line["cpu_baseline"] = {"value": round(ms, 1), "unit": "ms", "cores": cores,
                                "kind": "oracle", "sample": sample}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


def max_over_ranks(vals, dist, device):
    """Each value's maximum over the ranks (replicas: the job's TTFT is its
    slowest replica's); the values unchanged on a single process."""
    if dist is None:
        return [float(x) for x in vals]
    import torch
    t = torch.tensor([float(x) for x in vals], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t]


def run_sweep(r, args, rank):
    m = r.m
    pts = []
    for frac in r.sc["fractions"]:
        for pol in r.sc["policies"]:
            vals, comp, copy = [], [], []
            # per-kernel events only in the last warm-up step (they would
            # otherwise add to the timed steps)
            ks = {}
            for i in range(args.warmup + args.steps):
                m.mzc_set_kernel_timing(r.c, -1 if i == args.warmup - 1 else 0)
                r.evict(pol, frac)
                d, h, st, times = r.step()
                if i == args.warmup - 1:
                    ks = {nm: round(m.mzc_kernel_stats(r.c, j).ms, 3)
                          for j, nm in enumerate(m.KERNEL_CLASS_NAMES)}
                if i >= args.warmup:
                    vals.append(d)
                    comp.append(float(times[0]))
                    copy.append(float(times[1]))
            m.mzc_set_kernel_timing(r.c, 0)
            pt = {"fraction": frac, "policy": pol, "ttft_ms": round(statistics.median(vals), 3),
                  "p10": round(float(np.percentile(vals, 10)), 3),
                  "p90": round(float(np.percentile(vals, 90)), 3),
                  "compute_stream_ms": round(statistics.median(comp), 3),
                  "copy_stream_ms": round(statistics.median(copy), 3),
                  "kernel_ms": ks,
                  "recompute_rows": st.recompute_rows_last,
                  "copied_bytes": st.bytes_h2d_last if pol != "recompute" else 0}
            pts.append(pt)
            print(json.dumps(pt), file=sys.stderr, flush=True)
    if rank == 0:
        best = {}
        for p in pts:
            best.setdefault(p["fraction"], {})[p["policy"]] = p["ttft_ms"]
        print(json.dumps({"metric": METRIC, "workload": _describe("3b_sweep", r.sc), "swap_codec": args.codec,
                          "profile": {k: getattr(r.profile, k) for k, _ in r.profile._fields_},
                          "sweep": best, "points": pts}), flush=True)


def run_order(r, args, rank):
    """Eviction-order ablation (Sec. 6.3, Fig. 12b): the same number of whole
    layers (weights and every KV block) swapped out backward-out, forward-out or
    at random, restored forward-in while the prompt runs."""
    import synth
    m, L, N = r.m, r.shape["n_layers"], r.N
    res, pts = {}, []
    for frac in r.sc["fractions"]:
        k = int(round(frac * L))
        for order in r.sc["orders"]:
            if order == "backward":
                draws = [list(range(L - k, L))]
            elif order == "forward":
                draws = [list(range(k))]
            else:
                draws = [sorted(synth.permutation(synth.SEED_EVICT, 10 + d, L)[:k].tolist())
                         for d in range(r.sc["random_draws"])]
            vals = []
            for layers in draws:
                for i in range(args.warmup + args.steps):
                    for l in layers:
                        m.mzc_evict_weights(r.c, l, l + 1)
                        m.mzc_evict(r.c, l, l + 1, 0, N, m.MZC_COPY)
                    d, h, st, times = r.step()
                    if i >= args.warmup:
                        vals.append(d)
            pt = {"fraction": frac, "order": order, "layers_per_draw": k, "draws": len(draws),
                  "ttft_ms": round(statistics.median(vals), 3),
                  "p10": round(float(np.percentile(vals, 10)), 3),
                  "p90": round(float(np.percentile(vals, 90)), 3)}
            pts.append(pt)
            res.setdefault(frac, {})[order] = pt["ttft_ms"]
            print(json.dumps(pt), file=sys.stderr, flush=True)
    if rank == 0:
        print(json.dumps({"metric": "TTFT ms by eviction order", "workload": _describe("3b_order", r.sc),
                          "swap_codec": args.codec, "order": res, "points": pts}), flush=True)


def run_decode(r, args, rank):
    """Decode after the first token: greedy single-token steps over the
    resident context (each step is a one-row prefill through the same path)."""
    m, sh = r.m, r.shape
    tok = np.array([int(r.prompt[0])], np.int32)
    vals = []
    for i in range(args.warmup + args.steps):
        m.mzc_prefill(r.c, tok, r.logits)
        t = m.mzc_last_times(r.c)
        tok = np.array([int(np.argmax(r.logits))], np.int32)
        if i >= args.warmup:
            vals.append(float(t[3]))
    # one more step with every kernel class timed (not part of the median)
    m.mzc_set_kernel_timing(r.c, -1)
    m.mzc_prefill(r.c, tok, r.logits)
    ks = {nm: round(m.mzc_kernel_stats(r.c, j).ms, 4) for j, nm in enumerate(m.KERNEL_CLASS_NAMES)}
    m.mzc_set_kernel_timing(r.c, 0)
    m.mzc_truncate(r.c, r.N)
    ms = statistics.median(vals)
    d, hq, hkv, hd, L = (sh[k] for k in ("d_model", "n_q_heads", "n_kv_heads", "head_dim", "n_layers"))
    params = L * (d * (hq + 2 * hkv) * hd + hq * hd * d + 3 * d * sh["ffn_dim"]) + sh["vocab"] * d
    kv = L * r.N * 2 * hkv * hd * 2
    bytes_step = 2 * params + kv
    if rank == 0:
        print(json.dumps({"metric": "decode ms per token", "workload": _describe(r.name, r.sc),
                          "value": round(ms, 3), "unit": "ms", "tokens_per_s": round(1e3 / ms, 1),
                          "bytes_per_token": int(bytes_step),
                          "hbm_gbs": round(bytes_step / (ms * 1e-3) / 1e9, 1),
                          "kernel_ms_per_token": ks}), flush=True)


if __name__ == "__main__":
    main()
