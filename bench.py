"""Benchmark of KV-PRM verify-token scoring on GB300.

One step = one kvprm_score call: the verify token of every candidate in the
batch forwarded through all layers against its paged cache (embedding, per
layer RMSNorm / QKV / RoPE / paged split-K attention / combine / O / RMSNorm /
SiLU-gated MLP, final norm and the two-logit head).  Default workload: the
largest configuration that fits one GPU, the 8B-shaped scorer (32 layers,
d=4096, 32/8 heads, hd=128, MLP 14336) scoring B=8 candidates with distinct
caches of L=32768 (page size 16; 48.3 GB of weights and cache per call),
seeded synthetic bf16 weights N(0, 0.02) and K/V N(0, 1).

Printed (rank 0, one JSON line): scores/s over the timed steps with inputs
resident in HBM (`value`), the same through the host-buffer C-ABI call with
the cache copied host->device every step (`e2e`), the per-kernel-class CUDA
event times of a profiled pass, the time each kernel class adds to the
pipelined timeline of a traced call, the roofline of the dominant kernel and
of the attention, the SM clocks seen during the timed region, the CPU oracle
timed on a bounded sample of the same workload (`cpu_baseline`, with the
single-thread oracle on the two small configurations), and `workloads`: the
other four configurations measured the same way in the same run.

`--impl reference` times the CPU oracle alone (the reference arm).
Multi-GPU (torchrun): each rank scores its own replica batch (candidates
shard with no exchange), weak scaling, max time over ranks.
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import os
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

HBM_NOMINAL_GBS = 8000.0   # the 8 TB/s denominator the metric is quoted against
METRIC = "verify-token scores/sec"


def load_peaks() -> dict:
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "src": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "src": "fallback"}


# ---------------------------------------------------------------- distributed
def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch
        import torch.distributed as dist
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend=backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ---------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        # raw samples (the JSON line carries their summary); KVPRM_CLOCKS_DIR keeps them somewhere chosen
        out_dir = os.environ.get("KVPRM_CLOCKS_DIR") or tempfile.gettempdir()
        self.path = os.path.join(out_dir, f"clocks_rank{gpu_index}.csv")

    def start(self):
        os.makedirs(os.path.dirname(self.path), exist_ok=True)
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"], stdout=self.fh,
                                         stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.fh.close()
        sm, smax, reasons, power = [], [], set(), []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
                power.append(float(parts[3]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm), "power_w_max": max(power) if power else None}


# ---------------------------------------------------------------- workload
def algorithmic_bytes(w) -> dict:
    import kvsynth as ks
    a = w.arch
    per = {
        "gemm_qkv": a.n_layers * 2 * a.qkv_rows * a.d_model,
        "gemm_o": a.n_layers * 2 * a.d_model * a.n_q_heads * a.head_dim,
        "gemm_gate_up": a.n_layers * 2 * 2 * a.d_ff * a.d_model,
        "gemm_down": a.n_layers * 2 * a.d_model * a.d_ff,
        "attention": w.unique_kv_bytes(),
    }
    r = a.lora_rank
    if r:   # scorer adapter: each projection also streams B [out][r]; the A x launches stream A [r][in]
        per["gemm_qkv"] += a.n_layers * 2 * a.qkv_rows * r
        per["gemm_o"] += a.n_layers * 2 * a.d_model * r
        per["gemm_gate_up"] += a.n_layers * 2 * 2 * a.d_ff * r
        per["gemm_down"] += a.n_layers * 2 * a.d_model * r
        per["adapter"] = a.n_layers * 2 * r * (2 * a.d_model + a.n_q_heads * a.head_dim + a.d_ff)
    per["weights_total"] = a.weight_bytes()
    per["call_total"] = per["weights_total"] + per["attention"]
    del ks
    return per


def source_hash(files: list[str]) -> str:
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


KERNEL_SOURCES = {
    "gemm": ["paper_2607_09153_gb300/csrc/gemm_tc.cu", "paper_2607_09153_gb300/csrc/ptx.cuh",
             "paper_2607_09153_gb300/csrc/kernels.h"],
    "attention": ["paper_2607_09153_gb300/csrc/attention.cu", "paper_2607_09153_gb300/csrc/attn_core.cuh",
                  "paper_2607_09153_gb300/csrc/ptx.cuh", "paper_2607_09153_gb300/csrc/kernels.h"],
}


def ncu_traffic(kernel: str, workload: str):
    """Per-launch DRAM bytes from the committed ncu summary, if it was taken on
    the current kernel source (else None)."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
        e = rec[workload][kernel]
        fam = "gemm" if kernel.startswith("gemm") else "attention"
        if e.get("source_hash") != source_hash(KERNEL_SOURCES[fam]):
            return None
        return float(e["dram_bytes_per_launch"])
    except Exception:
        return None


# ---------------------------------------------------------------- CPU oracle
class OracleRunner:
    """The oracle (exact mode) on a fixed sample of a workload's candidates: weights and the sample's
    logical K/V are generated once, beforehand; one step scores the sample once."""

    def __init__(self, w, tables, nthreads: int | None = None, depth: int = 1):
        import kvsynth as ks
        self.w, self.tables, self.depth = w, tables, depth
        self.nthreads = nthreads or (os.cpu_count() or 1)
        t0 = time.perf_counter()
        self.W = ks.host_weights(w.arch, w.seed, tables)
        self.t_gen = time.perf_counter() - t0
        self.kv = {}

    def step(self, ids) -> float:
        import kvsynth as ks
        import oracle
        a = self.w.arch
        for b in ids:
            if b not in self.kv:
                self.kv[b] = [ks.host_kv_logical(self.w, l, b, self.tables) for l in range(a.n_layers)]
        kv = [[self.kv[b][l] for b in ids] for l in range(a.n_layers)]
        t = time.perf_counter()
        oracle.score_dense(a, self.W, kv, mirror=False, want_attn=False, nthreads=self.nthreads, depth=self.depth)
        return time.perf_counter() - t

    def sample_size(self, budget_s: float) -> int:
        """Candidates per step so that one step takes about budget_s (at least one)."""
        t1 = self.step([0])
        return int(max(1, min(self.w.n_candidates, budget_s / max(t1, 1e-3))))

    def describe(self, n: int, t: float, steps: int = 1) -> str:
        return (f"{n} of {self.w.n_candidates} candidates of {self.w.name} per step, fp64 exact mode, "
                f"{t:.2f} s per step over {steps} step(s), {self.nthreads} thread(s) (weights generated "
                f"beforehand in {self.t_gen:.1f} s and the sample's K/V before the first step, not timed)")


def cpu_oracle_time(w, tables, budget_s: float = 12.0, depth: int = 1, nthreads: int | None = None):
    """The oracle timed on a bounded sample of the workload's candidates (the first n)."""
    r = OracleRunner(w, tables, nthreads, depth)
    n = r.sample_size(budget_s)
    t = r.step(list(range(n)))
    return {"value": n / t, "unit": "scores/s", "cores": r.nthreads, "kind": "oracle", "sample": r.describe(n, t)}


def run_reference(args, world, rank):
    """The reference arm: the CPU oracle as it stands, on this host's cores.  One step scores a fixed
    sample of the workload's candidates, sized by the rule the main arm's cpu_baseline uses (about
    --cpu-budget of work, or ~--ref-step-s per step when given); ms_per_step is that observed step
    time and value the sample's candidates per second."""
    if rank != 0:
        return
    import kvsynth as ks
    w = make_workload(args)
    t = ks.Tables.make()
    runner = OracleRunner(w, t, depth=args.depth)
    n = runner.sample_size(args.ref_step_s if args.ref_step_s > 0 else args.cpu_budget)
    ids = list(range(n))
    times = []
    for i in range(args.warmup + args.steps):
        dt = runner.step(ids)
        if i >= args.warmup:
            times.append(dt)
    step_s = float(np.mean(times))
    val = n / step_s
    line = {"impl": "reference", "metric": METRIC, "value": val, "unit": "scores/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * step_s,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": dict(workload_config(w, args), reference_step=f"{n} of {w.n_candidates} candidates"),
            "cpu_baseline": {"value": val, "unit": "scores/s", "cores": runner.nthreads, "kind": "oracle",
                             "sample": runner.describe(n, step_s, args.steps)},
            "e2e": {"value": val, "unit": "scores/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def make_workload(args, name: str | None = None):
    """The named workload (--workload unless `name` is given); with --lora R its scorer carries an
    adapter of rank R (alpha 32) apart from the merged weights (every projection y = W x + (alpha / R)
    B (A x)); with --layers N the same shapes with N layers (small profiler captures)."""
    import dataclasses
    import kvsynth as ks
    w = ks.make_workload(name or args.workload)
    if args.lora:
        w.arch = dataclasses.replace(w.arch, lora_rank=args.lora)
    if args.layers:
        w.arch = dataclasses.replace(w.arch, n_layers=args.layers)
    return w


def workload_config(w, args) -> dict:
    a = w.arch
    return {"workload": w.name, "layers": a.n_layers, "d_model": a.d_model, "n_q_heads": a.n_q_heads,
            "n_kv_heads": a.n_kv_heads, "head_dim": a.head_dim, "d_ff": a.d_ff, "candidates": w.n_candidates,
            "seq_len_min": int(w.seq_lens.min()), "seq_len_max": int(w.seq_lens.max()), "page_size": a.page_size,
            "unique_pages": unique_pages(w),
            "l2": "inputs exceed L2 (weights + cache >> 129 MB); no flush", "parallelism": f"replicas{args.gpus}",
            **({"lora_rank": a.lora_rank, "lora_alpha": a.lora_alpha} if a.lora_rank else {}),
            **({"readout_depth": args.depth} if args.depth > 1 else {})}


def unique_pages(w) -> int:
    return int(len(set(np.concatenate([w.block_table[b, :(int(w.seq_lens[b]) + 15) // 16]
                                       for b in range(w.n_candidates)]).tolist())))


# ---------------------------------------------------------------- GPU arm
def make_scorer(dev, max_candidates: int, max_blocks: int):
    import kvsynth as ks
    from paper_2607_09153_gb300 import Scorer
    a = dev.arch
    wt = {"embed_verify": dev.top[ks.EMBED], "final_norm": dev.top[ks.FINAL_NORM], "w_plus": dev.top[ks.W_PLUS],
          "w_minus": dev.top[ks.W_MINUS],
          "layers": [{"attn_norm": L[ks.ATTN_NORM], "w_qkv": L[ks.W_QKV], "w_o": L[ks.W_O], "mlp_norm": L[ks.MLP_NORM],
                      "w_gate_up": L[ks.W_GATE_UP], "w_down": L[ks.W_DOWN],
                      **({"q_norm": L[ks.Q_NORM], "k_norm": L[ks.K_NORM]} if a.qk_norm else {})} for L in dev.layers]}
    sc = Scorer(a.n_layers, a.d_model, a.n_q_heads, a.n_kv_heads, a.head_dim, a.d_ff, wt, max_candidates, max_blocks,
                a.rope_base, a.rms_eps, qk_norm=a.qk_norm)
    if a.lora_rank:   # the scorer adapter, kept apart from the base weights
        names = dict(zip(ks.LORA_KINDS, ("a_qkv", "b_qkv", "a_o", "b_o", "a_gate_up", "b_gate_up", "a_down", "b_down")))
        sc.set_lora(a.lora_rank, a.lora_alpha, [{names[k]: L[k] for k in ks.LORA_KINDS} for L in dev.layers])
    return sc


def measure(w, args, world, local, steps: int, warmup: int, prof_steps: int, with_e2e: bool, clocks: bool):
    """Time one workload: K scoring calls (kvprm_score_async, graph replay) with inputs resident in HBM,
    then (with_e2e) the host-buffer call with the cache copied in every step, then a profiled pass
    (per-kernel-class CUDA events, launch overlap off) and one traced call (device timeline, launch
    overlap kept).  Returns a dict of measurements."""
    import torch

    import kvsynth as ks
    import paper_2607_09153_gb300 as kp

    tables = ks.Tables.make()
    dev = ks.DeviceInputs(w, tables)
    a = w.arch
    B = w.n_candidates
    sc = make_scorer(dev, B * args.depth, w.max_blocks)
    if args.depth > 1:   # depth-k readout: k verify tokens per candidate, rows of the same batch
        sc.set_depth(args.depth)
    stream = torch.cuda.Stream()
    sp = stream.cuda_stream
    d_rewards = torch.empty(B, dtype=torch.float32, device="cuda")
    pool_ptr, n_pages = dev.pool.data_ptr(), dev.n_pages
    bt, sl = np.ascontiguousarray(w.block_table), np.ascontiguousarray(w.seq_lens)

    def step():
        kp.kvprm_score_async(sc.ctx, pool_ptr, n_pages, bt, sl, B, d_rewards.data_ptr(), sp)

    for _ in range(warmup):
        step()
    stream.synchronize()
    clk = ClockSampler(local) if clocks else None
    barrier(world)
    torch.cuda.synchronize()
    if clk:
        clk.start()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(steps):
        step()
    ev1.record(stream)
    ev1.synchronize()
    torch.cuda.synchronize()
    barrier(world)
    clk_rec = clk.stop() if clk else None
    ms = max_over_ranks(ev0.elapsed_time(ev1), world)
    kp.kvprm_check_device(sc.ctx)
    # host side of one call (validation, attention schedule, table upload, graph launch), each call
    # made with the GPU idle so that no wait for an earlier call's staging buffer is counted
    host_s = []
    for _ in range(5):
        stream.synchronize()
        t0 = time.perf_counter()
        step()
        host_s.append(time.perf_counter() - t0)
    stream.synchronize()
    out = {"ms": ms, "steps": steps, "clocks": clk_rec, "host_us_per_call": round(1e6 * float(np.median(host_s)), 1)}
    # the attention schedule alone, as the call builds it (kvprm_plan_attention, host only)
    share = 3 if a.head_dim == 128 else 1
    tp = time.perf_counter()
    for _ in range(5):
        kp.kvprm_plan_attention(w.block_table, w.seq_lens, a.n_kv_heads, a.n_q_heads // a.n_kv_heads,
                                torch.cuda.get_device_properties(0).multi_processor_count, share | kp.KVPRM_PLAN_FUSE)
    out["plan_us"] = round(1e6 * (time.perf_counter() - tp) / 5, 1)

    if with_e2e:   # end to end through the host-buffer call (cache copied H2D every step)
        host_pool = torch.empty(dev.pool.shape, dtype=dev.pool.dtype, pin_memory=True)
        host_pool.copy_(dev.pool)
        rewards = np.zeros(B, np.float32)
        e2e_steps = max(3, steps // 10)
        for _ in range(2):
            kp.kvprm_score_host(sc.ctx, host_pool.data_ptr(), n_pages, bt, sl, B, sp, rewards)
        barrier(world)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(e2e_steps):
            kp.kvprm_score_host(sc.ctx, host_pool.data_ptr(), n_pages, bt, sl, B, sp, rewards)
        t_e2e = max_over_ranks(time.perf_counter() - t0, world)
        h2d = int(host_pool.numel() * 2 + bt.nbytes + sl.nbytes)
        out["e2e"] = {"value": world * B * e2e_steps / t_e2e, "unit": "scores/s",
                      "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": int(B * 4 + 4), "steps": e2e_steps,
                      # host->device bytes moved per second inside the timed region (the host link's
                      # ~211 GB/s bounds it: the call is copy-bound)
                      "h2d_gbs": round(h2d * e2e_steps / t_e2e / 1e9, 1),
                      "path": "kvprm_score_host: pinned host cache + host tables -> rewards on host"}
        del host_pool

    # per-kernel-class CUDA event times (launch overlap off, each launch timed alone)
    kp.kvprm_set_profile(sc.ctx, True)
    for _ in range(prof_steps):
        step()
    out["prof"] = kp.kvprm_get_profile(sc.ctx)
    kp.kvprm_set_profile(sc.ctx, False)
    stream.synchronize()
    # one traced call: each launch's first-CTA start and last-CTA end with launch overlap kept
    kp.kvprm_set_trace(sc.ctx, True)
    step()
    out["trace"] = kp.kvprm_get_trace(sc.ctx)
    kp.kvprm_set_trace(sc.ctx, False)
    stream.synchronize()
    sc.close()
    del dev
    torch.cuda.empty_cache()
    return out


def pipelined_times(trace, n_layers: int) -> dict:
    """Per kernel class, the time it adds to the call's timeline: from the later of its own start and
    the previous launch's end to its own end (launch overlap kept), summed, per layer."""
    tot = {}
    prev_end = None
    for cls, t0, t1 in trace:
        begin = t0 if prev_end is None else max(t0, prev_end)
        tot[cls] = tot.get(cls, 0.0) + max(0.0, t1 - begin)
        prev_end = t1 if prev_end is None else max(prev_end, t1)
    return {k: round(v / n_layers, 3) for k, v in tot.items()}


def summarize(w, m: dict, world: int) -> dict:
    """Rooflines and rates of one measured workload."""
    a = w.arch
    B = w.n_candidates
    prof = m["prof"]
    alg = algorithmic_bytes(w)
    peaks = load_peaks()
    prof_steps = max(1, max(n for n, _ in prof.values()) // max(1, a.n_layers)) if prof else 1
    kernels = {}
    for name, (n, tot) in prof.items():
        if n:
            kernels[name] = {"launches": n, "total_ms": round(tot, 4), "avg_us": round(1000 * tot / n, 3)}
    total_ms = sum(k["total_ms"] for k in kernels.values()) or 1.0
    for k in kernels.values():
        k["share"] = round(k["total_ms"] / total_ms, 4)
    n_calls = prof.get("gemm_qkv", (0, 0))[0] // a.n_layers or 1
    layers_timed = n_calls * a.n_layers
    classes = {"attention": ("attention", "attention_tc")}
    piped = pipelined_times(m["trace"], a.n_layers)

    def roof(name):
        parts = [c for c in classes.get(name, (name,)) if prof.get(c, (0, 0.0))[0] > 0]
        n = sum(prof[c][0] for c in parts)
        tot = sum(prof[c][1] for c in parts)
        per_layer = alg[name] / a.n_layers
        layer_s = tot / layers_timed / 1000.0
        ach = per_layer / layer_s / 1e9
        pip_us = sum(piped.get(c, 0.0) for c in parts)
        return {"bound": "hbm", "achieved": round(ach, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": round(ach / peaks["hbm_gbs"], 4), "peak_src": peaks["src"],
                "frac_of_8tbs": round(ach / HBM_NOMINAL_GBS, 4),
                "traffic": ncu_traffic(name, w.name) if len(parts) == 1 else None, "kernel": "+".join(parts),
                "algorithmic_bytes_per_launch": int(per_layer), "launches_per_layer": round(n / layers_timed, 3),
                "avg_launch_us": round(1000.0 * tot / n, 3), "time_per_layer_us": round(layer_s * 1e6, 3),
                "pipelined_us_per_layer": round(pip_us, 3) if pip_us else None,
                "pipelined_frac": round(per_layer / (pip_us * 1e-6) / 1e9 / peaks["hbm_gbs"], 4) if pip_us else None}

    cand = [k for k in kernels if k in alg or k == "attention_tc"]
    dominant = max((k for k in cand if k in alg), key=lambda k: kernels[k]["total_ms"]
                   + (kernels.get("attention_tc", {}).get("total_ms", 0.0) if k == "attention" else 0.0))
    attn = roof("attention")
    call_s = m["ms"] / m["steps"] / 1000.0
    logical = w.logical_kv_bytes()
    kv_tok = a.kv_bytes_per_token()
    # with the combine (the split partials' merge) counted in the attention step's time
    comb_n, comb_ms = prof.get("combine", (0, 0.0))
    attn_comb_s = (attn["time_per_layer_us"] * 1e-6 + comb_ms / layers_timed / 1000.0) if comb_n else None
    attention_obj = {"achieved_gbs": attn["achieved"], "frac_of_8tbs": attn["frac_of_8tbs"],
                     "with_combine": {"time_per_layer_us": round(attn_comb_s * 1e6, 3),
                                      "frac_of_8tbs": round(alg["attention"] / a.n_layers / attn_comb_s / 1e9
                                                            / HBM_NOMINAL_GBS, 4)} if attn_comb_s else
                     {"time_per_layer_us": attn["time_per_layer_us"], "frac_of_8tbs": attn["frac_of_8tbs"],
                      "note": "combine inside the attention launch (fused plan)"},
                     "frac_of_measured": attn["frac"], "unique_kv_bytes_per_step": alg["attention"],
                     "logical_kv_bytes_per_step": int(logical),
                     "logical_gbs": round(logical / a.n_layers / (attn["time_per_layer_us"] * 1e-6) / 1e9, 1),
                     "time_per_layer_us": attn["time_per_layer_us"], "kernels": attn["kernel"],
                     "pipelined_us_per_layer": attn["pipelined_us_per_layer"],
                     "pipelined_frac_of_8tbs": round(alg["attention"] / a.n_layers / (attn["pipelined_us_per_layer"]
                                                      * 1e-6) / 1e9 / HBM_NOMINAL_GBS, 4)
                     if attn["pipelined_us_per_layer"] else None}
    step_bytes = alg["call_total"]
    return {
        "scores_per_s": round(world * B / call_s, 2), "ms_per_call": round(call_s * 1e3, 5),
        "us_per_call": round(call_s * 1e6, 2),
        "kv_tokens_per_s": {"logical": round(logical / kv_tok / call_s, 1),
                            "unique": round(alg["attention"] / kv_tok / call_s, 1)},
        "whole_call": {"bytes_per_step": step_bytes, "achieved_gbs": round(step_bytes / call_s / 1e9, 1),
                       "frac_of_8tbs": round(step_bytes / call_s / 1e9 / HBM_NOMINAL_GBS, 4),
                       "frac_of_measured": round(step_bytes / call_s / 1e9 / peaks["hbm_gbs"], 4)},
        "attention": attention_obj, "roofline": roof(dominant), "kernels": kernels,
        "pipelined_us_per_layer": piped,
        "host": {"us_per_call": m["host_us_per_call"], "plan_us": m["plan_us"]},
        "launches_per_call": int(round(sum(n for n, _ in prof.values()) / max(1, n_calls))),
        "profile_steps": prof_steps,
    }


OTHER_WORKLOADS = ("tiny", "qwen1p5b_b16_l2048", "beam7b_b64_p4096_s512", "mcts7b_b256_d4")


def run_steering_only(args, world, rank, local):
    """The KV Steering gradient alone on --workload (the case ncu captures of the backward use)."""
    import torch
    torch.cuda.set_device(local)
    line = measure_steering(args, args.workload, calls=args.steps, warmup=args.warmup)
    line["metric"] = "KV Steering gradient calls/s"
    if rank == 0:
        print(json.dumps(line), flush=True)


def measure_steering(args, name: str, calls: int = 5, warmup: int = 1) -> dict:
    """KV Steering's gradient (kvprm_score_grad: the forward with its intermediates kept, then the
    backward into every referenced page) on one workload: blocking calls timed on the host clock.
    Algorithmic bytes per call: the weights twice (forward, then their transposes), the unique K/V
    twice (forward and backward reads) and the gradient written in fp32 (twice the K/V bytes)."""
    import torch

    import kvsynth as ks
    import paper_2607_09153_gb300 as kp
    w = make_workload(args, name)
    t = ks.Tables.make()
    dev = ks.DeviceInputs(w, t)
    sc = make_scorer(dev, w.n_candidates, w.max_blocks)
    grad = torch.empty(dev.pool.shape, dtype=torch.float32, device="cuda")
    st = torch.cuda.current_stream().cuda_stream
    args_ = (sc.ctx, dev.pool.data_ptr(), dev.n_pages, w.block_table, w.seq_lens, w.n_candidates, grad.data_ptr(), st)
    t0 = time.perf_counter()
    kp.kvprm_score_grad(*args_)   # the first call also builds the transposed weights
    first_s = time.perf_counter() - t0
    for _ in range(warmup):
        kp.kvprm_score_grad(*args_)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(calls):
        kp.kvprm_score_grad(*args_)
    call_s = (time.perf_counter() - t0) / calls
    alg = algorithmic_bytes(w)
    step_bytes = 2 * alg["weights_total"] + 4 * alg["attention"]
    peaks = load_peaks()
    sc.close()
    del grad, dev
    torch.cuda.empty_cache()
    return {"workload": name, "entry_point": "kvprm_score_grad", "grad_calls_per_s": round(1.0 / call_s, 2),
            "ms_per_call": round(call_s * 1e3, 3), "first_call_ms": round(first_s * 1e3, 1),
            "algorithmic_bytes_per_call": int(step_bytes),
            "achieved_gbs": round(step_bytes / call_s / 1e9, 1),
            "frac_of_measured": round(step_bytes / call_s / 1e9 / peaks["hbm_gbs"], 4), "calls": calls,
            "timing": "blocking calls on the host clock (the call synchronises)"}


def run_gpu(args, world, rank, local):
    import torch
    import kvsynth as ks
    torch.cuda.set_device(local)
    w = make_workload(args)
    m = measure(w, args, world, local, args.steps, args.warmup, args.profile_steps, with_e2e=True, clocks=True)
    sm = summarize(w, m, world)
    line = {
        "metric": METRIC, "value": round(world * w.n_candidates * args.steps / (m["ms"] / 1000.0), 2),
        "unit": "scores/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(m["ms"] / args.steps, 5), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "accumulate": "f32",
        "data": "synthetic (seeded bf16 weights N(0,0.02), K/V N(0,1), random-init)",
        "config": workload_config(w, args),
        "e2e": m["e2e"],
        "gpu_launches": sm["launches_per_call"] * args.steps,
        "roofline": sm["roofline"],
        "attention": sm["attention"],
        "whole_call": sm["whole_call"],
        "kv_tokens_per_s": sm["kv_tokens_per_s"],
        "host": sm["host"],
        "kernels": sm["kernels"],
        "pipelined_us_per_layer": sm["pipelined_us_per_layer"],
        "profile_steps": sm["profile_steps"],
        "clocks": m["clocks"],
    }
    # the other configurations, measured the same way in the same run (shorter timed regions)
    if world == 1 and not args.no_workloads and not args.layers and not args.lora and args.depth == 1:
        line["workloads"] = {}
        for name in OTHER_WORKLOADS:
            if name == w.name:
                continue
            wo = make_workload(args, name)
            mo = measure(wo, args, world, local, min(args.steps, 20), 3, 3, with_e2e=False, clocks=True)
            so = summarize(wo, mo, world)
            entry = {k: so[k] for k in ("scores_per_s", "ms_per_call", "kv_tokens_per_s", "whole_call", "host",
                                        "launches_per_call", "pipelined_us_per_layer")}
            entry["kernel_avg_us"] = {k: v["avg_us"] for k, v in so["kernels"].items()}
            if name == "tiny":
                entry["us_per_call"] = so["us_per_call"]
            else:
                entry["attention"] = {k: so["attention"][k] for k in ("achieved_gbs", "frac_of_8tbs", "frac_of_measured",
                                                                     "time_per_layer_us", "pipelined_us_per_layer",
                                                                     "pipelined_frac_of_8tbs", "with_combine",
                                                                     "kernels")}
                entry["roofline"] = so["roofline"]
            entry["config"] = workload_config(wo, args)
            entry["clocks"] = mo["clocks"]
            line["workloads"][name] = entry
        if not args.no_steering:
            line["steering"] = measure_steering(args, "qwen1p5b_b16_l2048")
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        tables = ks.Tables.make()
        line["cpu_baseline"] = cpu_oracle_time(w, tables, budget_s=args.cpu_budget, depth=args.depth)
        if not args.layers and not args.lora and args.depth == 1:   # single-thread oracle on the two small configs
            one = {}
            for name, budget in (("tiny", 2.0), ("qwen1p5b_b16_l2048", 4.0)):
                one[name] = cpu_oracle_time(make_workload(args, name), tables, budget_s=budget, nthreads=1)
            line["cpu_baseline"]["single_thread"] = one
    if rank == 0:
        print(json.dumps(line), flush=True)


def run_attention_only(args, world, rank, local):
    """The paged attention read-out alone (kvprm_attention: split-K attention
    plus combine) on ONE layer of the workload's cache, timed per kernel with
    CUDA events; a few-GB footprint, the case ncu captures use."""
    import dataclasses

    import torch

    import kvsynth as ks
    import paper_2607_09153_gb300 as kp

    torch.cuda.set_device(local)
    w = make_workload(args)
    a = w.arch
    # the workload's heads and cache on a one-layer scorer (its projections are never run here)
    w1 = dataclasses.replace(w, arch=ks.Arch(1, 256, a.n_q_heads, a.n_kv_heads, a.head_dim, 256, a.rope_base,
                                             a.rms_eps))
    dev = ks.DeviceInputs(w1, ks.Tables.make())
    B = w.n_candidates
    sc = make_scorer(dev, B, w.max_blocks)
    gen = torch.Generator(device="cuda")
    gen.manual_seed(7)
    q = torch.randn(B, a.n_q_heads, a.head_dim, device="cuda", generator=gen)
    kself = torch.randn(B, a.n_kv_heads, a.head_dim, device="cuda", generator=gen)
    vself = torch.randn(B, a.n_kv_heads, a.head_dim, device="cuda", generator=gen)
    out = torch.empty_like(q)
    stream = torch.cuda.Stream()
    bt, sl = np.ascontiguousarray(w.block_table), np.ascontiguousarray(w.seq_lens)

    def step():
        kp.kvprm_attention(sc.ctx, dev.pool[0].data_ptr(), dev.n_pages, bt, sl, B, q.data_ptr(), kself.data_ptr(),
                           vself.data_ptr(), out.data_ptr(), stream.cuda_stream)

    for _ in range(args.warmup):
        step()
    stream.synchronize()
    clocks = ClockSampler(local)
    clocks.start()
    kp.kvprm_set_profile(sc.ctx, True)
    for _ in range(args.steps):
        step()
    prof = kp.kvprm_get_profile(sc.ctx)
    kp.kvprm_set_profile(sc.ctx, False)
    clk = clocks.stop()
    kp.kvprm_check_device(sc.ctx)
    n_at, t_at = prof["attention"]
    n_tc, t_tc = prof["attention_tc"]   # shared pages on the tensor cores (a second launch per call)
    n_cb, t_cb = prof["combine"]
    kv_bytes = w.unique_kv_bytes() // a.n_layers   # one layer, each distinct page once
    at_s = (t_at + t_tc) / args.steps / 1000.0
    peaks = load_peaks()
    ach = kv_bytes / at_s / 1e9
    line = {
        "metric": "paged attention HBM GB/s (one layer, kernel time)", "value": round(ach, 1), "unit": "GB/s",
        "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "higher_is_better": True, "dtype": "bf16",
        "data": "synthetic (seeded K/V N(0,1); random fp32 q / self k / self v)",
        "config": dict(workload_config(w, args), layers=1,
                       l2="one layer's cache; inputs larger than L2 except small workloads, no flush"),
        "roofline": {"bound": "hbm", "achieved": round(ach, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
                     "frac": round(ach / peaks["hbm_gbs"], 4), "peak_src": peaks["src"],
                     "frac_of_8tbs": round(ach / HBM_NOMINAL_GBS, 4), "traffic": ncu_traffic("attention", w.name) if not n_tc else None,
                     "kernel": "attention" + ("+attention_tc" if n_tc else ""),
                     "algorithmic_bytes_per_launch": int(kv_bytes), "time_per_call_us": round(at_s * 1e6, 3),
                     "launches_per_call": (n_at + n_tc) / args.steps,
                     "tc_share": round(t_tc / (t_at + t_tc), 4) if n_tc else 0.0},
        "combine_avg_us": round(1000 * t_cb / max(n_cb, 1), 3),
        "clocks": clk,
    }
    sc.close()
    if rank == 0:
        print(json.dumps(line), flush=True)


def main():
    import kvsynth as ks
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="long8b_b8_l32768", choices=list(ks.WORKLOAD_NAMES))
    ap.add_argument("--no-workloads", action="store_true",
                    help="measure the --workload alone (by default the other configurations follow, shorter)")
    ap.add_argument("--ref-step-s", type=float, default=0.0,
                    help="reference arm: candidates per step chosen so that one step takes about this long "
                         "(0, the default: the --cpu-budget rule, so the arm times the cpu_baseline's sample)")
    ap.add_argument("--depth", type=int, default=1,
                    help="verify tokens per candidate (depth-k readout; 1, the default: one)")
    ap.add_argument("--layers", type=int, default=0,
                    help="run the workload's shapes with this many layers (0: all; for small profiler captures)")
    ap.add_argument("--lora", type=int, default=0,
                    help="scorer adapter rank kept apart from the weights (0: merged weights, the default)")
    ap.add_argument("--profile-steps", type=int, default=5)
    ap.add_argument("--cpu-budget", type=float, default=12.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-steering", action="store_true", help="skip the KV Steering gradient measurement")
    ap.add_argument("--steering-only", action="store_true",
                    help="time the KV Steering gradient (kvprm_score_grad) alone on --workload")
    ap.add_argument("--attention-only", action="store_true",
                    help="time the paged attention alone on one layer of the workload's cache")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    world, rank, local = dist_setup()
    if args.impl == "reference":
        run_reference(args, world, rank)
    elif args.attention_only:
        run_attention_only(args, world, rank, local)
    elif args.steering_only:
        run_steering_only(args, world, rank, local)
    else:
        run_gpu(args, world, rank, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
