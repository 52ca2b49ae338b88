#!/usr/bin/env python3
"""Benchmark: time-to-first-token of restoration-overlapped prefill on GB300.

One step = one TTFT: mzc_restore_async -> mzc_recompute_tail -> mzc_prefill
(prompt) -> first-token logits in host memory, over a context whose evicted
part was put back at rest (evicted) before the step, outside the timed region
(the paper's TTFT includes restoration but not eviction, Sec. 6.1).

Default (no --workload): the metric's lead, TTFT vs evicted fraction on the
3B-class model (3b_sweep: 32768-token context, 128-token prompt, evicted
token-tail fraction f in {0, 10, 25, 50, 75, 100}% x {copy, recompute,
hybrid}).  `value` is the hybrid TTFT at f = 1 (the whole context evicted);
every (fraction, policy) point is in `sweep` / `points`.  The same run then times the 1B-class
recompute workload (recompute tok/s and % of the BF16 tensor peak, the
metric's other two parts) under `recompute_1b`.

Other workloads (--workload, one line each; synthetic stand-ins for the
paper's models, see synth/workloads.py):
  1b_recompute            16L d2048, 8192-token context, tail [4096, 8192)
                          dropped and recomputed, 128-token prompt
  tiny                    2L d256, 512-token context, tail 256 dropped, 32-token prompt
  3b_scattered_copy       28L d3072, 32768-token context, 30% of blocks swapped to
                          pinned host and copied back while the prompt (256) runs
  3b_mixed                28L, last 8 layers' weights streamed, tail >= 16384 dropped,
                          20% of the rest copied, 512-token prompt
  3b_order, 1b_decode, 3b_decode   ablation / decode lines

value: device TTFT (CUDA events: start of the restore copies, or of the prefill when
nothing is copied, to the logits landing in host memory), median over the timed steps.
e2e: the same TTFT on the host clock through the C ABI with host buffers.
--impl reference: the CPU oracle (the repo's plain fp32 restatement) timed on a
bounded sample of the same workload's rows, scaled to the whole step.
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
    """Per-launch DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum)
    from the committed ncu capture of this kernel class on this workload, or
    None when there is none or the kernel's source changed since the counters
    were taken."""
    import hashlib
    try:
        with open(os.path.join(ROOT, "profiles", "ncu_traffic.json")) as f:
            entries = json.load(f)["entries"]
        for t in entries:
            if t.get("class") != kernel_class or t.get("workload") != workload:
                continue
            src = open(os.path.join(ROOT, t["source"]), "rb").read()
            if hashlib.sha256(src).hexdigest()[:16] != t["source_sha"]:
                return None
            return t["bytes_per_launch"]
    except Exception:
        return None
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
    if name == "3b_sweep":
        return (f"{name}: {base}, evicted token-tail fraction x restore policy (copy / recompute / "
                f"hybrid), {sc['prompt']}-token prompt")
    return f"{name}: {base}"


class Runner:
    """Owns one ctx on one GPU and knows how to put the evicted state at rest
    (untimed) and run one timed restore + prefill."""

    def __init__(self, name, sc, device, codec=0, read_swapped=0, wait_mode=0, separate_norm=0,
                 fused_rope=0):
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
        self.c = m.mzc_create(sh, self.w, max_rows=max_rows, device=device, swap_codec=codec,
                              read_swapped=read_swapped, wait_mode=wait_mode,
                              separate_norm=separate_norm, fused_rope=fused_rope)
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


# the 3B sweep point reported as `value`: the whole context evicted (the
# largest restore, where copy and recompute are balanced against each other)
HEADLINE = (1.0, "hybrid")


def _config(name, sc, codec, n_gpus, wait_mode="event", separate_norm=False, fused_rope=False):
    """The `config` object; both arms print the same one."""
    cfg = {"workload": _describe(name, sc), "swap_codec": codec, "wait_mode": wait_mode,
           "rmsnorm": "separate launches" if separate_norm else "folded into the projections at 1 and 5-256 rows",
           "rope_kv_write": "inside the QKV projection at 5-256 rows" if fused_rope else "its own launch",
           "l2": "inputs larger than L2 (weights + KV >> 129 MB)",
           "parallelism": f"replicas x{n_gpus}" if n_gpus > 1 else "single GPU",
           "timed": "restore + recompute + prompt prefill + logits D2H per step; eviction between steps untimed"}
    if name == "3b_sweep":
        cfg["value_point"] = {"fraction": HEADLINE[0], "policy": HEADLINE[1]}
        cfg["fractions"] = list(sc["fractions"])
        cfg["policies"] = list(sc["policies"])
    return cfg


def _cpu_model():
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    import platform
    return platform.machine()


_ORACLE_CACHE = {}


def _oracle_rows(name, sc):
    """Positions the oracle computes for one step of the workload, and the KV
    bytes its restore copies.  The oracle restores exactly (copy = memcpy of
    the evicted bytes, or recompute of a dropped tail as a prefill of those
    rows): for the 3B sweep it takes the copy path for the whole evicted tail,
    its fastest exact restore, and then prefills the prompt."""
    sh = sc["model"]
    N, P = sc["context"], sc["prompt"]
    kv_token = 2 * sh["n_layers"] * sh["n_kv_heads"] * sh["head_dim"] * 2
    if "evict_tail" in sc:
        rec, copy_bytes = sc["evict_tail"], 0
    elif "drop_from" in sc:
        rec = N - sc["drop_from"]
        copy_bytes = int(round(sc["scatter_frac"] * sc["drop_from"])) * kv_token
    elif name == "3b_scattered_copy":
        rec, copy_bytes = 0, int(round(sc["scatter_frac"] * N)) * kv_token
    elif name == "3b_sweep":
        rec = 0
        copy_bytes = int(np.ceil(HEADLINE[0] * (N // 16))) * 16 * kv_token
    else:
        rec, copy_bytes = 0, 0
    pos = np.concatenate([np.arange(N - rec, N), np.arange(N, N + P)]).astype(np.int64)
    return pos, copy_bytes


def _oracle_setup(sc):
    import oracle
    import synth
    sh = sc["model"]
    key = tuple(sorted((k, v) for k, v in sh.items())) + (sc["context"], sc["prompt"])
    if key not in _ORACLE_CACHE:
        _ORACLE_CACHE.clear()
        w = synth.model_weights(sh)
        ctx_len = sc["context"] + sc["prompt"]
        kv = oracle.KVState.__new__(oracle.KVState)
        dims = (sh["n_layers"], ctx_len, sh["n_kv_heads"], sh["head_dim"])
        kv.k = np.zeros(dims, np.float32)   # KV-conditioned state: the resident context
        kv.v = np.zeros(dims, np.float32)
        kv.max_ctx = ctx_len
        _ORACLE_CACHE[key] = (w, kv)
    return _ORACLE_CACHE[key]


def _memcpy_ms(nbytes):
    """Host memcpy time of nbytes, from a timed 256 MiB copy (the oracle's
    copy restore: swapped bytes back into its KV state)."""
    if nbytes <= 0:
        return 0.0
    n = 256 << 20
    a = np.ones(n, np.uint8)
    b = np.empty_like(a)
    np.copyto(b, a)
    t = time.perf_counter()
    np.copyto(b, a)
    dt = time.perf_counter() - t
    return dt * 1e3 * nbytes / n


def _oracle_step(name, sc, idx):
    """Times the oracle on rows idx (indices into the step's row list) through
    every layer over the KV-conditioned state, plus the LM head of one row and
    the restore copy; returns (ms scaled to the whole step, wall s, rows)."""
    import oracle
    import synth
    sh = sc["model"]
    pos, copy_bytes = _oracle_rows(name, sc)
    w, kv = _oracle_setup(sc)
    idx = np.asarray(idx, dtype=np.int64)
    toks = synth.tokens(synth.SEED_PROMPT, 9, idx.size, sh["vocab"])
    t0 = time.perf_counter()
    oracle.forward(sh, w, kv, toks, pos[idx], logits=False)
    t_rows = time.perf_counter() - t0
    x = np.ones((1, sh["d_model"]), np.float32)
    t = time.perf_counter()
    h = oracle.rmsnorm(x, w["final_norm"], sh["rms_eps"])
    oracle.linear(h, w["lm_head"])
    t_lm = time.perf_counter() - t
    copy_ms = _memcpy_ms(copy_bytes)
    ms = t_rows * 1e3 * pos.size / idx.size + t_lm * 1e3 + copy_ms
    return ms, time.perf_counter() - t0 + copy_ms * 1e-3, pos.size


def _sample_note(name, sc, n_rows, total, extra=""):
    sh = sc["model"]
    _, copy_bytes = _oracle_rows(name, sc)
    rows = (f"all {total} rows of the step (unsampled)" if n_rows >= total else
            f"{n_rows} of {total} rows (evenly spaced over the step's recomputed tail and prompt)")
    scale = "" if n_rows >= total else f", scaled x{total / n_rows:.1f} (extrapolated)"
    return (f"{rows} through all {sh['n_layers']} layers over a KV-conditioned state of "
            f"{sc['context'] + sc['prompt']} positions{scale}, "
            f"plus one LM-head row and a host memcpy of the {copy_bytes / 1e9:.2f} GB the step restores "
            f"by copy{extra}")


def cpu_baseline(name, sc, full=False):
    """The oracle on the GPU machine's host cores: 4 x cores rows of the step
    (every core busy), or every row with `full` (minutes at 1B scale), a
    1-thread time on 2 rows, the CPU model, and the tiny workload run
    unsampled."""
    import oracle
    oracle.build()
    cores = oracle.num_threads()
    pos, _ = _oracle_rows(name, sc)
    # the tiny workload runs whole (a small sample would be mostly per-call cost)
    n = pos.size if (name == "tiny" or full) else min(pos.size, 4 * cores)
    idx = np.unique(np.linspace(0, pos.size - 1, n).astype(int))
    ms, wall, total = _oracle_step(name, sc, idx)
    oracle.set_num_threads(1)
    try:
        idx1 = np.unique(np.linspace(0, pos.size - 1, min(2, pos.size)).astype(int))
        ms1, wall1, _ = _oracle_step(name, sc, idx1)
    finally:
        oracle.set_num_threads(cores)
    from synth import workloads as W
    tiny = dict(W.SCENARIOS["tiny"])
    tpos, _ = _oracle_rows("tiny", tiny)
    tiny_ms, _, _ = _oracle_step("tiny", tiny, np.arange(tpos.size))
    _ORACLE_CACHE.clear()
    return {"value": round(ms, 1), "unit": "ms", "cores": cores, "kind": "oracle",
            "sample": _sample_note(name, sc, idx.size, total, f"; {wall:.1f} s of wall time"),
            "cpu_model": _cpu_model(),
            "one_thread": {"value": round(ms1, 1), "unit": "ms", "threads": 1,
                           "sample": f"{idx1.size} of {total} rows, scaled likewise; {wall1:.1f} s of wall time"},
            "tiny_unsampled_ms": round(tiny_ms, 2)}


def run_reference(args, name, sc, rank):
    """The reference arm: the CPU oracle as it stands, each timed step one
    bounded sample of the workload's rows (one row per core, a different
    evenly spread slice each step, so the K steps together cover K x cores
    rows), scaled to the whole step.  Warm-up steps run one row each.
    ms_per_step is the wall time a sampled step actually took; value is the
    median of the scaled whole-step TTFTs."""
    if rank != 0:
        return
    import oracle
    oracle.build()
    cores = oracle.num_threads()
    pos, _ = _oracle_rows(name, sc)
    total = pos.size
    per = total if name == "tiny" else min(total, cores)
    order = np.argsort((np.arange(total) * 0.6180339887) % 1.0, kind="stable")  # spread slices
    vals, walls = [], []
    for i in range(args.warmup):
        _oracle_step(name, sc, order[:1])
    for i in range(args.steps):
        sl = order[(i * per) % total: (i * per) % total + per]
        if sl.size < per:
            sl = np.concatenate([sl, order[: per - sl.size]])
        ms, wall, _ = _oracle_step(name, sc, np.sort(sl))
        vals.append(ms)
        walls.append(wall)
    v = statistics.median(vals)
    line = {"impl": "reference", "metric": METRIC, "value": round(v, 3), "unit": "ms",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(statistics.mean(walls) * 1e3, 3), "higher_is_better": False,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": _config(name, sc, args.codec, args.gpus, args.wait_mode, args.separate_norm, args.fused_rope),
            "extrapolated": {"rows_per_timed_step": int(per), "rows_per_step": int(total),
                             "note": "value scales each step's sampled rows to the whole step; "
                                     "ms_per_step is the sampled step's own wall time"},
            "cpu_baseline": {"value": round(v, 3), "unit": "ms", "cores": cores, "kind": "oracle",
                             "sample": _sample_note(name, sc, per, total, "; a different slice each step"),
                             "cpu_model": _cpu_model()},
            "e2e": {"value": round(v, 3), "unit": "ms", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


ROOFLINE_NOTE = ("dominant class's launches bracketed by CUDA events on the compute stream over "
                 "K further steps of the same workload, run right after the K timed steps "
                 "(the timed steps carry no events)")


def _roofline(ks, dom, peaks, src, workload):
    if ks is None:
        return None
    k = ks[dom]
    if k.ms <= 0 or k.launches <= 0:
        return None
    per = k.launches
    # the bound follows the launches' arithmetic intensity: below the ridge
    # (sustained FLOP/s over HBM bytes/s) a contraction streams its operands
    ridge = peaks["bf16_tflops_sustained"] * 1e12 / (peaks["hbm_gbs"] * 1e9)
    tensor_bound = dom in ("gemm", "attention") and (k.bytes <= 0 or k.flops / k.bytes >= ridge)
    if tensor_bound:
        ach = k.flops / (k.ms * 1e-3) / 1e12
        peak = peaks["bf16_tflops_sustained"]
        return {"kernel": dom, "bound": "tensor", "achieved": round(ach, 2), "peak": peak,
                "unit": "TFLOP/s", "frac": round(ach / peak, 4), "traffic": _traffic(dom, workload),
                "measured_over": ROOFLINE_NOTE,
                "peak_source": f"{src} bf16 sustained (fp16 operands: nominal fp16/bf16 ratio 1.0)",
                "frac_of_burst": round(ach / peaks["bf16_tflops"], 4),
                "avg_launch_ms": round(k.ms / per, 4), "flops_per_launch": k.flops / per,
                "launches": int(per)}
    ach = k.bytes / (k.ms * 1e-3) / 1e9
    peak = peaks["hbm_gbs"]
    return {"kernel": dom, "bound": "hbm", "achieved": round(ach, 1), "peak": peak,
            "unit": "GB/s", "frac": round(ach / peak, 4), "traffic": _traffic(dom, workload),
            "measured_over": ROOFLINE_NOTE,
            "peak_source": f"{src} HBM copy", "avg_launch_ms": round(k.ms / per, 4),
            "bytes_per_launch": k.bytes / per, "launches": int(per)}


def _class_stats(m, c):
    return {nm: m.mzc_kernel_stats(c, i) for i, nm in enumerate(m.KERNEL_CLASS_NAMES)}


def _timed_workload(r, args, dist, name, evict, roofline=True):
    """W warm-up steps (the last one times every kernel class to find the
    dominant one), then exactly K timed steps bracketed by a barrier and a
    device synchronize, with no CUDA events between kernels (an event between
    two launches breaks their programmatic-dependent-launch overlap, which at
    ~10 us kernels moves the TTFT by up to 20%).  With `roofline`, K further
    steps of the same workload follow, with the dominant class's launches
    bracketed by CUDA events on the compute stream: its live per-launch time
    for the roofline; those steps are not part of the TTFT.  Returns per-step
    device and host TTFTs and the stats."""
    import torch
    m = r.m
    for i in range(args.warmup):
        m.mzc_set_kernel_timing(r.c, -1 if i == args.warmup - 1 else 0)
        evict()
        r.step()
    warm = _class_stats(m, r.c)
    dom = max(warm, key=lambda nm: warm[nm].ms)
    m.mzc_set_kernel_timing(r.c, 0)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    dev, host, comp, copy, st = [], [], [], [], None
    for _ in range(args.steps):
        evict()
        d, h, st, times = r.step()
        dev.append(d)
        host.append(h)
        comp.append(float(times[0]))
        copy.append(float(times[1]))
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    launches = _class_stats(m, r.c)  # counted with timing off
    ks = None
    if roofline and not args.no_kernel_timing:
        m.mzc_set_kernel_timing(r.c, 1 << m.KERNEL_CLASS_NAMES.index(dom))
        for _ in range(args.steps):
            evict()
            r.step()
        torch.cuda.synchronize()
        ks = _class_stats(m, r.c)
        m.mzc_set_kernel_timing(r.c, 0)
    return dict(dev=dev, host=host, comp=comp, copy=copy, st=st, warm=warm, dom=dom, ks=ks,
                launches=launches)


def _h2d_bytes(sc, st):
    sh = sc["model"]
    return int(st.rows_last * 8 + sh["n_layers"] * (-(-sh["max_ctx"] // 16)) * 4 + sc["prompt"] * 4
               + st.bytes_h2d_last)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="mzc", choices=["mzc", "reference"])
    ap.add_argument("--workload", default="3b_sweep",
                    choices=["3b_sweep", "1b_recompute", "tiny", "3b_scattered_copy", "3b_mixed",
                             "3b_order", "1b_decode", "3b_decode", "3b_read_swapped", "link",
                             "kernels", "projections"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-full", action="store_true",
                    help="time the oracle on every row of the step, unsampled (about 4 minutes "
                         "for 1b_recompute on 16 cores), instead of a 4 x cores-row sample")
    ap.add_argument("--no-kernel-timing", action="store_true")
    ap.add_argument("--no-1b", action="store_true", help="3b_sweep: skip the 1B recompute keys")
    ap.add_argument("--fractions", default=None, help="comma list overriding the sweep's fractions")
    ap.add_argument("--policies", default=None, help="comma list overriding the sweep's policies")
    ap.add_argument("--profile", default=None,
                    help="3b_sweep: the per-unit profile as 9 comma-separated numbers in "
                         "mzc_profile's field order (h2d_gbs, gemm_us_128, gemm_us_512, "
                         "gemm_us_2048, attn_tflops, attn_row_ns, attn_prompt_tflops, row_ns, "
                         "layer_us), as a default line's `profile` prints them; used instead of "
                         "measuring it (a run under ncu would plan from its own serialised "
                         "kernel times)")
    ap.add_argument("--profile-json", default=None,
                    help="3b_sweep: load the per-unit profile from this file if it exists, else "
                         "measure it and save it there")
    ap.add_argument("--wait-mode", default="event", choices=["event", "flag"],
                    help="how attention waits for restored blocks: per-layer events, or per-block "
                         "residency flags (MZC_WAIT_BLOCK_FLAG)")
    ap.add_argument("--codec", default="none", choices=["none", "q8"],
                    help="swap codec of the pinned store: none, or 8-bit groups (q8)")
    ap.add_argument("--separate-norm", action="store_true",
                    help="ablation: every RMSNorm as its own launch (no fold into the projections "
                         "for row sets of 1 or 5-256 rows)")
    ap.add_argument("--fused-rope", action="store_true",
                    help="the rotary embedding and KV-block write inside the QKV projection for row "
                         "sets of 5-256 rows (option fused_rope; measured no faster)")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "mzc":
        args.warmup = 3

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    name = args.workload
    if name in ("link", "kernels", "projections"):
        import torch
        if not torch.cuda.is_available():
            raise SystemExit("bench.py needs a CUDA GPU")
        import __graft_entry__
        __graft_entry__.build()
        {"link": run_link, "kernels": run_kernels, "projections": run_projections}[name](args)
        return
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

    r = Runner(name, sc, local, codec=1 if args.codec == "q8" else 0,
               read_swapped=1 if name == "3b_read_swapped" else 0,
               wait_mode=1 if args.wait_mode == "flag" else 0,
               separate_norm=1 if args.separate_norm else 0,
               fused_rope=1 if args.fused_rope else 0)
    if name == "3b_sweep":
        run_headline(r, args, rank, world, local, dist)
        if dist:
            dist.destroy_process_group()
        return
    if name == "3b_order":
        run_order(r, args, rank)
        r.close()
        return
    if name == "3b_read_swapped":
        run_read_swapped(r, args, rank)
        r.close()
        return
    if name.endswith("_decode"):
        run_decode(r, args, rank)
        r.close()
        return
    clk = Clocks(local)
    t_all = time.perf_counter()
    res = _timed_workload(r, args, dist, name, r.evict)
    wall = time.perf_counter() - t_all
    clocks = clk.stop()
    line = _single_line(r, args, world, name, sc, res, dist, clocks, wall)
    r.close()
    del r
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(name, sc, args.cpu_full)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


def _single_line(r, args, world, name, sc, res, dist, clocks, wall):
    v, e2e = max_over_ranks([statistics.median(res["dev"]), statistics.median(res["host"])], dist, "cuda")
    peaks, src = _peaks()
    ks, warm, st = res["ks"], res["warm"], res["st"]
    # launches of the library's kernels in the timed steps: the counted
    # classes plus one metadata-copy kernel per prefill call
    launches = sum(k.launches for k in res["launches"].values()) + args.steps
    roof = _roofline(ks, res["dom"], peaks, src, name)
    rows, rec_rows = st.rows_last, st.recompute_rows_last
    g, a = warm["gemm"], warm["attention"]
    gemm_tfs = g.flops / (g.ms * 1e-3) / 1e12 if g.ms > 0 else None
    attn_tfs = a.flops / (a.ms * 1e-3) / 1e12 if a.ms > 0 else None
    return {
        "metric": METRIC, "value": round(v, 3), "unit": "ms", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(statistics.mean(res["dev"]), 3), "higher_is_better": False,
        "scaling": "weak", "vs_baseline": None, "dtype": "f16",
        "data": "synthetic (seeded N(0,0.02) bf16 weights, uniform token ids)",
        "config": _config(name, sc, args.codec, world, args.wait_mode, args.separate_norm, args.fused_rope),
        "recompute_tok_s": round(rec_rows / (v * 1e-3), 1) if rec_rows else None,
        "rows_per_step": rows,
        "gemm_tflops": round(gemm_tfs, 1) if gemm_tfs else None,
        "attention_tflops": round(attn_tfs, 1) if attn_tfs else None,
        "tensor_peak_frac_gemm": round(gemm_tfs / peaks["bf16_tflops_sustained"], 4) if gemm_tfs else None,
        "tensor_peak_frac_gemm_burst": round(gemm_tfs / peaks["bf16_tflops"], 4) if gemm_tfs else None,
        "tensor_peak_frac_attention_burst": round(attn_tfs / peaks["bf16_tflops"], 4) if attn_tfs else None,
        "kernel_ms_per_step": {n: round(k.ms, 3) for n, k in warm.items()},
        "kernel_ms_source": "last warm-up step, every class timed",
        "roofline": roof,
        "e2e": {"value": round(e2e, 3), "unit": "ms", "h2d_bytes_per_step": _h2d_bytes(sc, st),
                "d2h_bytes_per_step": int(sc["model"]["vocab"] * 4)},
        "gpu_launches": int(launches),
        "clocks": clocks,
        "wall_s_timed": round(wall, 2),
        "setup_s": {"weights": round(r.t_gen, 1), "create": round(r.t_create, 1),
                    "context_prefill": round(r.t_ctx, 2)},
    }


def run_headline(r, args, rank, world, local, dist):
    """The default line: the 3B sweep (every fraction x policy; the HEADLINE
    point is `value`), then the 1B recompute workload's keys."""
    import torch
    m = r.m
    sc, name = r.sc, r.name
    if args.profile:
        vals = [float(x) for x in args.profile.split(",")]
        if len(vals) != len(m.mzc_profile._fields_):
            raise SystemExit("--profile takes %d numbers" % len(m.mzc_profile._fields_))
        r.profile = m.mzc_profile(*vals)
        m.mzc_set_policy(r.c, m.MZC_POLICY_HYBRID, r.profile)
    elif args.profile_json and os.path.exists(args.profile_json):
        # a profile saved by an earlier run (an ncu run would otherwise plan
        # from its own serialised kernel times)
        with open(args.profile_json) as f:
            d = json.load(f)
        r.profile = m.mzc_profile(*[float(d[k]) for k, _ in m.mzc_profile._fields_])
        m.mzc_set_policy(r.c, m.MZC_POLICY_HYBRID, r.profile)
    else:
        r.profile = m.mzc_profile_measure(r.c)
        if args.profile_json:
            with open(args.profile_json, "w") as f:
                json.dump({k: getattr(r.profile, k) for k, _ in r.profile._fields_}, f)
    peaks, src = _peaks()
    clk = Clocks(local)
    t_all = time.perf_counter()
    pts, head = [], None
    # the value point: HEADLINE, or the first point when --fractions /
    # --policies leave it out (a partial sweep, e.g. for a profiler run)
    grid = [(f, p) for f in sc["fractions"] for p in sc["policies"]]
    vp = HEADLINE if HEADLINE in grid else grid[0]
    for frac in sc["fractions"]:
        for pol in sc["policies"]:
            is_head = (frac, pol) == vp
            # the value point also takes the roofline steps; every point times
            # its kernel classes in the last warm-up step
            res = _timed_workload(r, args, dist if is_head else None, name,
                                  lambda: r.evict(pol, frac), roofline=is_head)
            st = res["st"]
            cp = statistics.median(res["copy"]) if pol != "recompute" and st.bytes_h2d_last else None
            pt = {"fraction": frac, "policy": pol, "ttft_ms": round(statistics.median(res["dev"]), 3),
                  "p10": round(float(np.percentile(res["dev"], 10)), 3),
                  "p90": round(float(np.percentile(res["dev"], 90)), 3),
                  "e2e_ms": round(statistics.median(res["host"]), 3),
                  "compute_stream_ms": round(statistics.median(res["comp"]), 3),
                  "copy_stream_ms": round(cp, 3) if cp else None,
                  "copied_bytes": int(st.bytes_h2d_last) if pol != "recompute" else 0,
                  "copy_gbs": round(st.bytes_h2d_last / (cp * 1e-3) / 1e9, 1) if cp else None,
                  "recompute_rows": int(st.recompute_rows_last),
                  "kernel_ms_warmup": {nm: round(k.ms, 3) for nm, k in res["warm"].items()}}
            pts.append(pt)
            print(json.dumps(pt), file=sys.stderr, flush=True)
            if is_head:
                head = res
    wall = time.perf_counter() - t_all
    sweep = {}
    for p in pts:
        sweep.setdefault(str(p["fraction"]), {})[p["policy"]] = p["ttft_ms"]
    vs = {}
    for f, d in sweep.items():
        if {"copy", "recompute", "hybrid"} <= set(d):
            vs[f] = {"hybrid_over_copy": round(d["hybrid"] / d["copy"], 4),
                     "hybrid_over_recompute": round(d["hybrid"] / d["recompute"], 4)}
    prof = {k: round(getattr(r.profile, k), 3) for k, _ in r.profile._fields_}
    line_extra = {}
    if head is not None:
        st = head["st"]
        cp = statistics.median(head["copy"])
        line_extra["restore_copy"] = {
            "bytes_per_step": int(st.bytes_h2d_last), "copy_stream_ms": round(cp, 3),
            "achieved_gbs": round(st.bytes_h2d_last / (cp * 1e-3) / 1e9, 1) if cp > 0 else None,
            "link_gbs_measured": round(r.profile.h2d_gbs, 1),
            "frac": round(st.bytes_h2d_last / (cp * 1e-3) / 1e9 / r.profile.h2d_gbs, 4) if cp > 0 else None,
            "link_source": "pinned host -> HBM copies timed by mzc_profile_measure in this process"}
    r.close()
    del r
    res1b = None
    if not args.no_1b:
        from synth import workloads as W
        r1 = Runner("1b_recompute", dict(W.SCENARIOS["1b_recompute"]), local)
        res1b = _timed_workload(r1, args, dist, "1b_recompute", r1.evict)
        l1 = _single_line(r1, args, world, "1b_recompute", r1.sc, res1b, dist, None, 0.0)
        r1.close()
        del r1
    clocks = clk.stop()
    v, e2e = max_over_ranks([statistics.median(head["dev"]), statistics.median(head["host"])], dist, "cuda")
    st = head["st"]
    line = {
        "metric": METRIC, "value": round(v, 3), "unit": "ms", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(statistics.mean(head["dev"]), 3), "higher_is_better": False,
        "scaling": "weak", "vs_baseline": None, "dtype": "f16",
        "data": "synthetic (seeded N(0,0.02) bf16 weights, uniform token ids)",
        "config": {**_config(name, sc, args.codec, world, args.wait_mode, args.separate_norm, args.fused_rope),
                   "value_point": {"fraction": vp[0], "policy": vp[1]}},
        "sweep": sweep, "hybrid_vs_policies": vs, "points": pts, "profile": prof,
        "roofline": _roofline(head["ks"], head["dom"], peaks, src, name),
        **line_extra,
        "e2e": {"value": round(e2e, 3), "unit": "ms", "h2d_bytes_per_step": _h2d_bytes(sc, st),
                "d2h_bytes_per_step": int(sc["model"]["vocab"] * 4)},
        "gpu_launches": int(sum(k.launches for k in head["launches"].values()) + args.steps),
        "gpu_launches_note": "the value point's timed steps: counted kernel classes plus one metadata-copy kernel per step",
        "kernel_ms_per_step": {nm: round(k.ms, 3) for nm, k in head["warm"].items()},
        "clocks": clocks,
        "clocks_span": "whole sweep and the 1B recompute steps",
        "wall_s_sweep": round(wall, 2),
    }
    if res1b is not None:
        line["recompute_1b"] = {k: l1[k] for k in (
            "value", "ms_per_step", "recompute_tok_s", "rows_per_step", "gemm_tflops",
            "attention_tflops", "tensor_peak_frac_gemm", "tensor_peak_frac_gemm_burst",
            "tensor_peak_frac_attention_burst", "kernel_ms_per_step", "roofline", "e2e", "gpu_launches")}
        line["recompute_1b"]["workload"] = l1["config"]["workload"]
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(name, sc, args.cpu_full)
    if rank == 0:
        print(json.dumps(line), flush=True)


def run_link(args):
    """Host-link probe (the copy path's per-unit rate, Sec. 4.3): pinned host
    -> HBM and HBM -> pinned host copy rates of 1 GiB with 1, 2, 4 and 8
    concurrent copy streams, with the NUMA node of the pinned pages and the
    GPU's NUMA affinity.  torch provides the pinned buffers and streams."""
    import ctypes
    import glob
    import torch
    G = 1 << 30
    h = torch.empty(G, dtype=torch.uint8, pin_memory=True)
    h.fill_(1)
    d = torch.empty(G, dtype=torch.uint8, device="cuda")
    libc = ctypes.CDLL(None, use_errno=True)
    page_node = None
    try:  # get_mempolicy(MPOL_F_NODE | MPOL_F_ADDR) on the first page
        nodev = ctypes.c_int(-1)
        nr = {"aarch64": 236, "x86_64": 239}.get(os.uname().machine)
        if nr and libc.syscall(nr, ctypes.byref(nodev), None, 0, ctypes.c_void_p(h.data_ptr()), 3) == 0:
            page_node = nodev.value
    except Exception:
        pass
    nodes = {}
    for pth in sorted(glob.glob("/sys/devices/system/node/node*/cpulist")):
        nodes[os.path.basename(os.path.dirname(pth))] = open(pth).read().strip()
    gpu_numa = None
    try:
        out = subprocess.run(["nvidia-smi", "topo", "-m"], capture_output=True, text=True, timeout=30).stdout
        for line in out.splitlines():
            if line.strip().startswith("GPU0") and "X" in line:
                gpu_numa = line.split()[-2] if len(line.split()) >= 4 else None
    except Exception:
        pass
    res = {"metric": "pinned host <-> HBM copy rate", "unit": "GB/s", "bytes": G,
           "numa_nodes": nodes, "pinned_page_node": page_node, "gpu_numa_affinity": gpu_numa}
    for k in (1, 2, 4, 8):
        streams = [torch.cuda.Stream() for _ in range(k)]
        sl = G // k
        for direction in ("h2d", "d2h"):
            best = 1e9
            for _ in range(max(3, args.steps)):
                torch.cuda.synchronize()
                t0 = time.perf_counter()
                for i, st in enumerate(streams):
                    with torch.cuda.stream(st):
                        if direction == "h2d":
                            d[i * sl:(i + 1) * sl].copy_(h[i * sl:(i + 1) * sl], non_blocking=True)
                        else:
                            h[i * sl:(i + 1) * sl].copy_(d[i * sl:(i + 1) * sl], non_blocking=True)
                torch.cuda.synchronize()
                best = min(best, time.perf_counter() - t0)
            res[f"{direction}_{k}_streams"] = round(G / best / 1e9, 1)
    print(json.dumps(res), flush=True)


def run_kernels(args):
    """The hot-path kernels one at a time through their C-ABI entry points:
    the two projection GEMM paths and the two attention kernels at the shapes
    listed below, and the memory-bound kernels at 3B-class shapes with inputs
    larger than L2 (129 MB): RMSNorm and the rotary/KV write over 16384 rows,
    the embedding gather over 16384 rows, the LM head over the 128256 x 3072
    bf16 head.  Per kernel: CUDA-event time per launch (median of the timed
    launches after warm-up), algorithmic bytes (and FLOPs) over that time,
    against the measured HBM copy rate (and BF16 peak).  About 2 GB of device
    memory in all: this is also the driver of the ncu captures of these
    kernels."""
    import torch
    import paper_2609_01338_gb300 as m
    peaks, src = _peaks()
    d, hq, hkv, hd, V, R = 3072, 24, 8, 128, 128256, 16384
    gen = torch.Generator(device="cuda").manual_seed(0)
    x = torch.randn((R, d), device="cuda", generator=gen)
    g = torch.ones(d, device="cuda")
    y = torch.empty((R, d), dtype=torch.int16, device="cuda")
    qkv = (torch.randn((R, (hq + 2 * hkv) * hd), device="cuda", generator=gen) * 0.5).half().view(torch.int16)
    pos = torch.arange(R, dtype=torch.int32, device="cuda")
    ang = torch.arange(R, dtype=torch.float64).unsqueeze(1) * (
        500000.0 ** (-2.0 * torch.arange(hd // 2, dtype=torch.float64) / hd)).unsqueeze(0)
    cos_t, sin_t = ang.cos().float().cuda(), ang.sin().float().cuda()
    n_logical = R // 16
    table = torch.randperm(n_logical, device="cuda", generator=gen).to(torch.int32)
    pool = torch.zeros((n_logical, 2, hkv, 16, hd), dtype=torch.int16, device="cuda")
    q_out = torch.empty((R, hq, hd), dtype=torch.int16, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    w_lm = (torch.randn((V, d), device="cuda", generator=gen) * 0.02).bfloat16().view(torch.int16)
    logits = torch.empty(V, device="cuda")
    emb = (torch.randn((V, d), device="cuda", generator=gen) * 0.02).bfloat16().view(torch.int16)
    toks = torch.randint(0, V, (R,), dtype=torch.int32, device="cuda", generator=gen)
    xe = torch.empty((R, d), device="cuda")
    # projections: the 3B down projection of a 128-row prompt (split-K cluster
    # GEMM, fp32 residual add) and the 1B gate/up projection of the 4224-row
    # recompute step (persistent GEMM, SwiGLU epilogue)
    a_sk = (torch.randn((128, 8192), device="cuda", generator=gen) * 0.5).half().view(torch.int16)
    w_sk = (torch.randn((d, 8192), device="cuda", generator=gen) * 0.02).half().view(torch.int16)
    o_sk = torch.zeros((128, d), device="cuda")
    M1, N1, K1 = 4224, 2 * 8192, 2048
    a_p = (torch.randn((M1, K1), device="cuda", generator=gen) * 0.5).half().view(torch.int16)
    w_p = (torch.randn((N1, K1), device="cuda", generator=gen) * 0.02).half().view(torch.int16)
    o_p = torch.empty((M1, N1 // 2), dtype=torch.int16, device="cuda")
    # attention: one 1B recompute-step layer (4224 rows at positions 4096..8319,
    # 32/8 heads of 64, tensor-core kernel) and one 3B decode token over 32768
    # keys (24/8 heads of 128, decode kernel); K/V in scattered blocks
    def attn_case(n_rows, ctx, hq_, hkv_, hd_, kvd):
        nl = -(-ctx // 16)
        tab = torch.randperm(nl, device="cuda", generator=gen).to(torch.int32)
        pl = (torch.randn((nl, 2, hkv_, 16, hd_), device="cuda", generator=gen)).half().view(torch.int16)
        q = (torch.randn((n_rows, hq_, hd_), device="cuda", generator=gen)).half().view(torch.int16)
        ps = torch.arange(ctx - n_rows, ctx, dtype=torch.int32, device="cuda")
        o = torch.empty_like(q)
        sb = m.mzc_k_attention_scratch_bytes(n_rows, hq_, hkv_, hd_, ctx)
        scr = torch.empty(max(sb, 16), dtype=torch.uint8, device="cuda")
        pairs = float(sum(range(ctx - n_rows + 1, ctx + 1)))
        fn = lambda: m.mzc_k_attention(q, ps, n_rows, hq_, hkv_, hd_, tab, nl, pl, nl, kvd, o, ctx,
                                       scr, sb, status)
        return fn, 4.0 * hd_ * hq_ * pairs, 2.0 * ctx * hkv_ * hd_ * 2 + 2.0 * n_rows * hq_ * hd_ * 2
    at_fn, at_fl, at_by = attn_case(4224, 8320, 32, 8, 64, 1)
    ad_fn, ad_fl, ad_by = attn_case(1, 32768, 24, 8, 128, 0)
    # the folded RMSNorm's two halves at the same 128 rows: the down projection
    # writing x * g and the per-tile sums of squares, then the QKV projection
    # (3072 -> 5120) scaling its rows by rstd
    h_sk = torch.empty((128, d), dtype=torch.int16, device="cuda")
    ss_sk = torch.zeros((128, d // 128), device="cuda")
    w_q = (torch.randn((5120, d), device="cuda", generator=gen) * 0.02).half().view(torch.int16)
    o_q = torch.empty((128, 5120), dtype=torch.int16, device="cuda")
    cases = {
        "gemm_splitk_kernel": (lambda: m.mzc_k_gemm(a_sk, w_sk, o_sk, 128, d, 8192, 1),
                               2.0 * (128 * 8192 + d * 8192) + 128 * d * 8.0, 2.0 * 128 * d * 8192),
        "gemm_splitk_kernel_norm_out": (
            lambda: m.mzc_k_gemm_norm_out(a_sk, w_sk, o_sk, 128, d, 8192, g, h_sk, ss_sk, status),
            2.0 * (128 * 8192 + d * 8192) + 128 * d * 10.0 + 128 * (d // 128) * 4.0, 2.0 * 128 * d * 8192),
        "gemm_splitk_kernel_norm_in": (
            lambda: m.mzc_k_gemm_norm_in(h_sk, w_q, o_q, 128, 5120, d, 0, ss_sk, 1e-5, status),
            2.0 * (128 * d + 5120 * d) + 128 * 5120 * 2.0 + 128 * (d // 128) * 4.0, 2.0 * 128 * 5120 * d),
        "gemm_persistent_kernel": (lambda: m.mzc_k_gemm(a_p, w_p, o_p, M1, N1, K1, 2),
                                   2.0 * (M1 * K1 + N1 * K1) + M1 * N1, 2.0 * M1 * N1 * K1),
        "attn_tc_kernel": (at_fn, at_by, at_fl),
        "attn_decode_kernel": (ad_fn, ad_by, ad_fl),
        "rmsnorm_warp_kernel": (lambda: m.mzc_k_rmsnorm(x, g, R, d, 1e-5, y), R * d * 6.0 + d * 4.0),
        "rope_kv_kernel": (lambda: m.mzc_k_rope_kv_write(qkv, pos, R, hq, hkv, hd, cos_t, sin_t, table,
                                                         n_logical, pool, n_logical, 0, q_out, status),
                           R * (hq + 2 * hkv) * hd * 4.0 + R * hd * 4.0),
        "embed_kernel": (lambda: m.mzc_k_embed(toks, R, emb, d, V, xe, status), R * d * 6.0),
        "lm_head_kernel": (lambda: m.mzc_k_lm_head(x[0], g, d, 1e-5, w_lm, V, logits),
                           V * d * 2.0 + V * 4.0 + d * 8.0),
    }
    out = {"metric": "hot-path kernels alone: algorithmic bytes (and FLOPs) over CUDA-event time",
           "peak_gbs": peaks["hbm_gbs"], "peak_source": f"{src} HBM copy",
           "shapes": f"d {d}, {hq}/{hkv} heads of {hd}, {R} rows, vocab {V}", "kernels": {}}
    for nm, case in cases.items():
        fn, nbytes, flops = case if len(case) == 3 else (*case, 0.0)
        for _ in range(max(3, args.warmup)):
            fn()
        torch.cuda.synchronize()
        ts = []
        for _ in range(max(5, args.steps)):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            fn()
            b.record()
            b.synchronize()
            ts.append(a.elapsed_time(b))
        ms = statistics.median(ts)
        k = {"ms": round(ms, 4), "bytes": int(nbytes), "gbs": round(nbytes / (ms * 1e-3) / 1e9, 1),
             "hbm_frac": round(nbytes / (ms * 1e-3) / 1e9 / peaks["hbm_gbs"], 4)}
        if flops:
            tf = flops / (ms * 1e-3) / 1e12
            k.update({"flops": flops, "tflops": round(tf, 1),
                      "tensor_frac_burst": round(tf / peaks["bf16_tflops"], 4)})
        out["kernels"][nm] = k
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    print(json.dumps(out), flush=True)


PROJECTIONS = {  # name: (rows, n, k, epilogue) of one decoder layer's projections
    "1b_qkv": (4224, 3072, 2048, 0), "1b_o": (4224, 2048, 2048, 1),
    "1b_gate_up": (4224, 16384, 2048, 2), "1b_down": (4224, 2048, 8192, 1),
    "3b_qkv": (2576, 5120, 3072, 0), "3b_o": (2576, 3072, 3072, 1),
    "3b_gate_up": (2576, 16384, 3072, 2), "3b_down": (2576, 3072, 8192, 1),
}


def run_projections(args):
    """The four projections of one decoder layer at the 1B recompute step's
    4224 rows and at the 3B value step's 2576 rows (hybrid, f = 1), one launch
    at a time through mzc_k_gemm: CUDA-event time per launch with L2 flushed
    before each (a 512 MB write), FLOPs over that time against the measured
    BF16 burst and sustained peaks.  Under 1.5 GB of device memory: also the
    driver of the ncu captures of the GEMM kernels (tensor-pipe activity per
    projection)."""
    import torch
    import paper_2609_01338_gb300 as m
    peaks, src = _peaks()
    flush = torch.empty(512 << 20, dtype=torch.uint8, device="cuda")
    gen = torch.Generator(device="cuda").manual_seed(0)
    out = {"metric": "prefill projections alone: FLOPs over CUDA-event time, L2 flushed before each launch",
           "peak_tflops_burst": peaks["bf16_tflops"], "peak_tflops_sustained": peaks["bf16_tflops_sustained"],
           "peak_source": src, "projections": {}}
    for name, (rows, n, k, epi) in PROJECTIONS.items():
        a = (torch.randn((rows, k), device="cuda", generator=gen) * 0.5).half().view(torch.int16)
        w = (torch.randn((n, k), device="cuda", generator=gen) * 0.02).half().view(torch.int16)
        o = (torch.zeros((rows, n), device="cuda") if epi == 1 else
             torch.empty((rows, n // 2 if epi == 2 else n), dtype=torch.int16, device="cuda"))
        ts = []
        for i in range(max(1, args.warmup) + max(1, args.steps)):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            m.mzc_k_gemm(a, w, o, rows, n, k, epi)
            e1.record()
            e1.synchronize()
            if i >= max(1, args.warmup):
                ts.append(e0.elapsed_time(e1))
        ms = statistics.median(ts)
        tf = 2.0 * rows * n * k / (ms * 1e-3) / 1e12
        out["projections"][name] = {
            "rows": rows, "n": n, "k": k, "us": round(ms * 1e3, 2), "tflops": round(tf, 1),
            "frac_sustained": round(tf / peaks["bf16_tflops_sustained"], 4),
            "frac_burst": round(tf / peaks["bf16_tflops"], 4)}
        del a, w, o
    # the 3B 128-row prompt: weight-streaming bound (the split-K cluster GEMM
    # for QKV, O and down, the persistent kernel for gate/up); each alone, and
    # one layer's four in sequence replayed from a CUDA graph (no host launch
    # cost; programmatic dependent launch between them), against the time to
    # stream the layer's 201 MB of weights at the measured HBM rate
    rows = 128
    d, q, f = 3072, 5120, 8192
    shapes = {"qkv": (q, d, 0), "o": (d, d, 1), "gate_up": (2 * f, d, 2), "down": (d, f, 1)}
    st = torch.cuda.Stream()
    bufs = {}
    for name, (n, k, epi) in shapes.items():
        a = (torch.randn((rows, k), device="cuda", generator=gen) * 0.5).half().view(torch.int16)
        w = (torch.randn((n, k), device="cuda", generator=gen) * 0.02).half().view(torch.int16)
        o = (torch.zeros((rows, n), device="cuda") if epi == 1 else
             torch.empty((rows, n // 2 if epi == 2 else n), dtype=torch.int16, device="cuda"))
        bufs[name] = (a, w, o, n, k, epi)
    def run_layer(stream):
        for a, w, o, n, k, epi in bufs.values():
            m.mzc_k_gemm(a, w, o, rows, n, k, epi, stream)
    prompt = {}
    for name, (a, w, o, n, k, epi) in bufs.items():
        ts = []
        for i in range(max(3, args.warmup) + max(5, args.steps)):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            m.mzc_k_gemm(a, w, o, rows, n, k, epi)
            e1.record()
            e1.synchronize()
            if i >= max(3, args.warmup):
                ts.append(e0.elapsed_time(e1))
        prompt[name] = {"n": n, "k": k, "us": round(statistics.median(ts) * 1e3, 2)}
    reps = 10
    with torch.cuda.stream(st):
        run_layer(st.cuda_stream)  # warm-up outside the capture
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=st):
            for _ in range(reps):
                run_layer(st.cuda_stream)
    ts = []
    for i in range(3 + max(5, args.steps)):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(st):  # the replay runs on the current stream
            e0.record(st)
            g.replay()
            e1.record(st)
        e1.synchronize()
        if i >= 3:
            ts.append(e0.elapsed_time(e1) / reps)
    wbytes = 2.0 * sum(n * k for _, _, _, n, k, _ in bufs.values())
    layer_us = statistics.median(ts) * 1e3
    out["prompt_3b_128_rows"] = {
        "projections_alone_us": prompt, "layer_graph_us": round(layer_us, 2),
        "weight_bytes": int(wbytes), "hbm_floor_us": round(wbytes / (peaks["hbm_gbs"] * 1e9) * 1e6, 2),
        "frac_of_hbm": round(wbytes / (layer_us * 1e-6) / (peaks["hbm_gbs"] * 1e9), 4)}
    print(json.dumps(out), flush=True)


def max_over_ranks(vals, dist, device):
    """Each value's maximum over the ranks (replicas: the job's TTFT is its
    slowest replica's); the values unchanged on a single process."""
    if dist is None:
        return [float(x) for x in vals]
    import torch
    t = torch.tensor([float(x) for x in vals], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t]


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


def run_read_swapped(r, args, rank):
    """Swapped blocks restored by copy (mzc_restore_async, then the prefill)
    against read in place by the attention kernels (the prefill alone, option
    read_swapped), for token tails of the 3B context (Sec. 4.2's shared
    buffers on a GB300: the same bytes cross the host link either way)."""
    m, L, N = r.m, r.shape["n_layers"], r.N
    res, pts = {}, []
    for frac in r.sc["fractions"]:
        p = max(0, N - int(np.ceil(frac * r.nblk)) * 16)
        for mode in ("copy", "in_place"):
            vals = []
            if mode == "in_place":
                m.mzc_evict(r.c, 0, L, p, N, m.MZC_COPY)  # stays swapped across the steps
            for i in range(args.warmup + args.steps):
                if mode == "copy":
                    m.mzc_evict(r.c, 0, L, p, N, m.MZC_COPY)
                    m.mzc_restore_async(r.c)
                m.mzc_prefill(r.c, r.prompt, r.logits)
                t = m.mzc_last_times(r.c)
                m.mzc_truncate(r.c, N)
                if i >= args.warmup:
                    vals.append(float(t[3]))
            if mode == "in_place":
                m.mzc_restore_async(r.c)
                m.mzc_sync(r.c)
            pt = {"fraction": frac, "mode": mode, "ttft_ms": round(statistics.median(vals), 3),
                  "p10": round(float(np.percentile(vals, 10)), 3),
                  "p90": round(float(np.percentile(vals, 90)), 3),
                  "swapped_bytes": int((N - p) * L * 2 * r.shape["n_kv_heads"] * r.shape["head_dim"] * 2)}
            pts.append(pt)
            res.setdefault(frac, {})[mode] = pt["ttft_ms"]
            print(json.dumps(pt), file=sys.stderr, flush=True)
    if rank == 0:
        print(json.dumps({"metric": "TTFT ms: swapped blocks copied back vs read in place",
                          "workload": _describe(r.name, r.sc), "ttft": res, "points": pts}), flush=True)


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
