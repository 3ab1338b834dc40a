"""Benchmark of the A-PACK inner-LLM prune step on GB300.

One benchmark step is one pass of the whole hot path over the workload: the
progressive schedule of the 7B-shaped 10-minute audio-video sequence
(135,272 tokens, 15,000 audio + 120,000 visual, 256 query rows, Hq 28 /
Hkv 4, pruning at layers 4, 12 and 20 of 28), i.e. three apack_prune_step
calls, each scoring, selecting and compacting K/V of all later layers and
the hidden states.  The metric is multimodal tokens entering the prune steps
per second (sum over steps of |S| / time).  The headline times the schedule
captured once into a CUDA graph (apack_prune_schedule_graph) and replayed per
step; the same JSON line carries the eager run (one apack_prune_schedule call
per step, with per-stage events), the end-to-end run with host buffers, and
the side measurements (the paper's own 14-step last-query setting, pre-LLM
alignment, decode attention).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Multi-GPU (torchrun): the step works on each sequence alone, so a batch of
several sequences splits over the ranks by whole sequences (strong scaling;
paper_2608_08794_gb300.shard), and a single sequence runs as one independent
replica per rank (weak scaling).  There is no data-path collective; the
barrier and max-over-ranks timing use torch.distributed, value = units of all
ranks / time.  ``--impl reference`` times the CPU oracle on a bounded sample
of the same workload (rank 0 only).
"""

import argparse
import hashlib
import json
import os
import platform
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "prune-step multimodal tokens/s; KV-compaction HBM GB/s vs peak (7B-shaped)"
UNIT = "multimodal tokens/s"
WORKLOAD = "7b_10min"
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS_SUSTAINED = 1700.0


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=200)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--workload", default=WORKLOAD)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--e2e-steps", type=int, default=None)
    p.add_argument("--replicas", action="store_true",
                   help="with several GPUs, run the whole batch on every rank instead of splitting its sequences")
    p.add_argument("--no-paper-setting", action="store_true",
                   help="skip the side measurement of the paper's own 14-step setting")
    p.add_argument("--part", default="all", choices=["all", "decode", "compact", "prellm"],
                   help="decode: time only the decode-step attention on a synthetic cache; compact: only "
                        "the first step's compaction of the 10-minute 7B cache, out of place and in place; "
                        "prellm: only the pre-LLM frame alignment of the workload's clip")
    p.add_argument("--window", type=int, default=3, help="prellm: the CKA window (odd, 1..7)")
    p.add_argument("--compact-planes", type=int, default=48,
                   help="compact: planes of 135272 rows (48 = K and V of layers 4..27)")
    p.add_argument("--decode-tokens", type=int, default=135272)
    p.add_argument("--decode-layers", type=int, default=8)
    return p.parse_args()


# ----------------------------------------------------------------------------- helpers

def max_over_ranks(x, dist, device):
    """The largest value of x over all ranks (x itself without a process group)."""
    if dist is None:
        return float(x)
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_value(units_per_rank, world, ms_per_iter):
    """Units of all ranks per second, each rank running its own replica."""
    return world * units_per_rank / (ms_per_iter / 1e3)


def sum_over_ranks(x, dist, device):
    """The sum of x over all ranks (x itself without a process group)."""
    if dist is None:
        return float(x)
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return float(d.get("hbm_gbs", FALLBACK_HBM_GBS)), "measured"
    return FALLBACK_HBM_GBS, "fallback"


def measured_tensor_peak():
    """Sustained dense bf16 TFLOP/s (for kernels timed inside a long step)."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        if "bf16_tflops_sustained" in d:
            return float(d["bf16_tflops_sustained"]), "measured (sustained)"
    return FALLBACK_BF16_TFLOPS_SUSTAINED, "fallback (sustained)"


def host_cpu():
    """CPU model and logical cores of this host."""
    model, arm = None, {}
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if ":" not in line:
                    continue
                key, val = (x.strip() for x in line.split(":", 1))
                if key.lower() in ("model name", "cpu model", "processor name") and model is None:
                    model = val
                elif key in ("CPU implementer", "CPU part") and key not in arm:
                    arm[key] = val
    except OSError:
        pass
    if model is None and arm:
        model = f"{platform.machine()} (implementer {arm.get('CPU implementer')}, part {arm.get('CPU part')})"
    return {"cpu_model": model or platform.processor() or platform.machine(), "nproc": os.cpu_count()}


GATHER_SOURCES = ["compact_tma.cu", "compact_plan.cuh"]   # the out-of-place gather and its item plan


def source_sha256(kernel_src):
    """sha256 of a kernel's source files (one name or a list, concatenated in order)."""
    names = [kernel_src] if isinstance(kernel_src, str) else list(kernel_src)
    h = hashlib.sha256()
    for n in names:
        with open(os.path.join(ROOT, "paper_2608_08794_gb300", "csrc", n), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def profiled_traffic(kernel_src, summary="gather_tma_traffic.json"):
    """DRAM bytes of a profiled launch from a committed ncu summary, if it was
    taken on the current kernel source (else None)."""
    path = os.path.join(ROOT, "profiles", summary)
    if not os.path.exists(path):
        return None
    with open(path) as f:
        d = json.load(f)
    if d.get("source_sha256") != source_sha256(kernel_src):
        return None
    return d


class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled every 100 ms."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.samples = []
        self.proc = None
        self.marks = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.samples.append((time.time(), line.strip()))

    def mark(self, on):
        self.marks.append((time.time(), on))

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        spans, t0 = [], None
        for t, on in self.marks:
            if on:
                t0 = t
            elif t0 is not None:
                spans.append((t0, t))
                t0 = None
        mhz, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for t, line in self.samples:
            if not any(a - 0.05 <= t <= b + 0.05 for a, b in spans):
                continue
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 7:
                continue
            try:
                mhz.append(float(parts[0]))
                mx = float(parts[1])
            except ValueError:
                continue
            for n, v in zip(names, parts[3:7]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not mhz:
            return {"sm_mhz": None, "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": 0}
        mhz.sort()
        return {"sm_mhz": mhz[len(mhz) // 2], "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(mhz)}


PAPER_CONTEXT = {
    "paper_prefill_flops_reduction": "up to 78% (Qwen2.5-Omni-7B, 25% tier, averaged over four benchmarks)",
    "paper_decode_throughput": "2.21x vs full tokens",
    "paper_hardware": "NVIDIA A6000 48 GB, bf16, FlashAttention-2, greedy decoding",
    "note": "the paper's end-to-end numbers, context only: they include the pre-LLM stage and the whole model",
}


def schedule_context(wl, pp):
    """The paper's headline numbers (context) and the analytic prefill-FLOPs ratio
    of the benchmarked inner-LLM schedule (App. G, single sequence; the pre-LLM
    stage is not part of this path)."""
    from paper_2608_08794_gb300 import flops as F
    ctx = dict(PAPER_CONTEXT)
    if wl.num_seqs != 1:
        return ctx
    model = F.QWEN25_OMNI_7B if wl.hidden == 3584 else F.QWEN25_OMNI_3B
    if wl.num_layers != model.layers:
        return ctx
    sched = F.layer_schedule(wl.total_tokens, list(zip(wl.prune_layers, pp.t_out)), model)
    ctx["inner_llm_prefill_flops_ratio"] = F.flops_ratio(sched, wl.total_tokens, model)
    ctx["inner_llm_note"] = "App. G accounting of this schedule alone (no pre-LLM compression)"
    return ctx


# ----------------------------------------------------------------------------- CPU oracle leg

ORACLE_SNIPPET = r"""
import json, sys, time
sys.path.insert(0, {root!r})
import numpy as np
import oracle
from synth import workload
from synth.configs import scaled_copy
from synth.inputs import query_rows, key_slab, value_slab, plain_key_slab, hidden_states, base_counts
wl = scaled_copy(workload({name!r}), {dur})
cu, cuq, mod = wl.cu_seqlens(), wl.cu_qlens(), wl.modality()
L, l0 = wl.num_layers, wl.prune_layers[0]
qs = [query_rows(wl, l) for l in wl.prune_layers]
ks = [key_slab(wl, l, q) for l, q in zip(wl.prune_layers, qs)]
# bulk K/V planes: one drawn layer repeated over the compacted layers (values do not change the copy cost)
kv = [np.repeat(plain_key_slab(wl, l0)[None], L - l0, axis=0), np.repeat(value_slab(wl, l0)[None], L - l0, axis=0)]
hid = hidden_states(wl)
if wl.joint_step_keep is None:
    counts = [oracle.step_keep_counts(r, base_counts(wl)) for r in wl.ratios]
else:
    counts, nS = [], [a + v for a, v in base_counts(wl)]
    for _ in wl.prune_layers:
        nS = [oracle.keep_count(wl.joint_step_keep, x) for x in nS]
        counts.append([(x, 0) for x in nS])
def one():
    comp = np.arange(wl.total_tokens); c, m = cu, mod
    kk, vv, hh = kv[0], kv[1], hid
    mm = 0
    for i, layer in enumerate(wl.prune_layers):
        mm += int(((m == 1) | (m == 2)).sum())
        j = layer - l0 if i == 0 else layer - wl.prune_layers[i - 1]
        out = oracle.prune_step(qs[i], ks[i][comp], c, cuq, m, wl.num_q_heads, wl.num_kv_heads, counts[i],
                                planes=[kk[j:].transpose(1, 0, 2, 3), vv[j:].transpose(1, 0, 2, 3), hh],
                                joint=wl.joint_step_keep is not None)
        keep = out["keep_idx"]
        kk = out["planes"][0].transpose(1, 0, 2, 3); vv = out["planes"][1].transpose(1, 0, 2, 3); hh = out["planes"][2]
        comp, c, m = comp[keep], out["cu_seqlens"], out["modality"]
    return mm, comp
reps = {reps}
times, mm = [], 0
for r in range(reps):
    t0 = time.perf_counter(); mm, comp = one(); times.append(time.perf_counter() - t0)
print(json.dumps(dict(times=times, mm=mm, tokens=wl.total_tokens, dur={dur}, kept=int(comp.size),
                      kept_sum=int(comp.sum()))))
"""


ORACLE_POOL_SNIPPET = r"""
import json, os, sys, time
sys.path.insert(0, {root!r})
import numpy as np
import multiprocessing as mp
from multiprocessing import shared_memory

_W = {{}}


def _attach(spec):
    shm = shared_memory.SharedMemory(name=spec[0])
    return shm, np.ndarray(spec[1], dtype=np.uint16, buffer=shm.buf)


def _init(specs, qs, mod, meta):
    import oracle
    _W["oracle"] = oracle
    _W["qs"], _W["mod"], _W["meta"] = qs, mod, meta
    for key, spec in specs.items():
        _W[key] = _attach(spec)


def _score(task):
    # the oracle's relevance scores of one KV head group and one chunk of query rows, weighted by
    # its share of the mean over all heads and rows (the mean is linear in its terms)
    i, g, r0, r1, comp, cu, mod = task
    oracle, hq, hkv, nq = _W["oracle"], _W["meta"]["hq"], _W["meta"]["hkv"], _W["meta"]["nq"]
    G = hq // hkv
    keys = _W["ks"][1][i][comp, g:g + 1]
    q = _W["qs"][i][r0:r1, g * G:(g + 1) * G]
    s = oracle.relevance_scores(q, keys, cu, np.array([0, r1 - r0], np.int32), mod, G, 1)
    return s * (G * (r1 - r0)) / float(hq * nq)


def _copy(task):
    kind, j, comp = task
    plane = _W[kind][1][j] if kind != "hid" else _W[kind][1]
    out = _W["oracle"].compact_rows(plane, comp)
    return int(out.shape[0])


if __name__ == "__main__":
    import oracle
    from synth import workload
    from synth.configs import scaled_copy
    from synth.inputs import query_rows, key_slab, value_slab, plain_key_slab, hidden_states, base_counts
    wl = scaled_copy(workload({name!r}), {dur})
    cu, cuq, mod = wl.cu_seqlens(), wl.cu_qlens(), wl.modality()
    L, l0, T = wl.num_layers, wl.prune_layers[0], wl.total_tokens
    qs = [query_rows(wl, l) for l in wl.prune_layers]
    arrays = {{"ks": np.stack([key_slab(wl, l, q) for l, q in zip(wl.prune_layers, qs)]),
              "kk": np.repeat(plain_key_slab(wl, l0)[None], L - l0, axis=0),
              "vv": np.repeat(value_slab(wl, l0)[None], L - l0, axis=0),
              "hid": hidden_states(wl)}}
    shms, specs = [], {{}}
    for key, a in arrays.items():
        shm = shared_memory.SharedMemory(create=True, size=a.nbytes)
        np.ndarray(a.shape, dtype=np.uint16, buffer=shm.buf)[...] = a
        shms.append(shm)
        specs[key] = (shm.name, a.shape)
    del arrays
    if wl.joint_step_keep is None:
        counts = [oracle.step_keep_counts(r, base_counts(wl)) for r in wl.ratios]
    else:
        counts, nS = [], [a + v for a, v in base_counts(wl)]
        for _ in wl.prune_layers:
            nS = [oracle.keep_count(wl.joint_step_keep, x) for x in nS]
            counts.append([(x, 0) for x in nS])
    nq = int(cuq[-1])
    meta = dict(hq=wl.num_q_heads, hkv=wl.num_kv_heads, nq=nq)
    workers = {workers}
    rows = max(1, -(-nq // max(1, (2 * workers) // wl.num_kv_heads)))
    ctx = mp.get_context("spawn")
    try:
        with ctx.Pool(workers, initializer=_init, initargs=(specs, qs, mod, meta)) as pool:
            pool.map(abs, range(4 * workers))            # every worker started and attached
            def one():
                comp, c, m = np.arange(T), cu, mod
                mm = 0
                for i, layer in enumerate(wl.prune_layers):
                    mm += int(((m == 1) | (m == 2)).sum())
                    tasks = [(i, g, r0, min(nq, r0 + rows), comp, c, m)
                             for g in range(wl.num_kv_heads) for r0 in range(0, nq, rows)]
                    scores = np.sum(pool.map(_score, tasks), axis=0)
                    keep = oracle.select_keep(scores, m, c, counts[i], joint=wl.joint_step_keep is not None)
                    comp, c, m = comp[keep], oracle.new_cu_seqlens(keep, c), oracle.compact_rows(m, keep)
                    # every later layer's K and V rows and the hidden states at the kept tokens
                    j0 = layer - l0
                    copies = [(kind, j, comp) for kind in ("kk", "vv") for j in range(j0, L - l0)]
                    pool.map(_copy, copies + [("hid", 0, comp)])
                return mm, comp
            one()                                         # warm-up: caches, page faults of the shared planes
            t0 = time.perf_counter()
            mm, comp = one()
            t = time.perf_counter() - t0
    finally:
        for shm in shms:
            shm.close()
            shm.unlink()
    print(json.dumps(dict(times=[t], mm=mm, tokens=T, dur={dur}, workers=workers, kept=int(comp.size),
                          kept_sum=int(comp.sum()))))
"""


def run_oracle_pool(name, dur, workers):
    """The oracle's schedule on `workers` processes: scoring split over (KV head group,
    query-row chunk), selection in the parent, the row copies split over planes."""
    env = dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1", MKL_NUM_THREADS="1")
    code = ORACLE_POOL_SNIPPET.format(root=ROOT, name=name, dur=dur, workers=workers)
    path = os.path.join("/tmp", f"apack_oracle_pool_{os.getpid()}.py")
    with open(path, "w") as f:
        f.write(code)
    try:
        r = subprocess.run([sys.executable, path], capture_output=True, text=True, env=env, cwd=ROOT)
    finally:
        os.remove(path)
    if r.returncode != 0:
        raise RuntimeError(r.stderr[-2000:])
    return json.loads(r.stdout.strip().splitlines()[-1])


def run_oracle(name, dur, reps):
    env = dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1", MKL_NUM_THREADS="1")
    code = ORACLE_SNIPPET.format(root=ROOT, name=name, dur=dur, reps=reps)
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env)
    if r.returncode != 0:
        raise RuntimeError(r.stderr[-2000:])
    return json.loads(r.stdout.strip().splitlines()[-1])


def cpu_sample_duration(name, budget_s, max_dur=360):
    """Clip length (even seconds) whose oracle schedule takes about budget_s."""
    probe = run_oracle(name, 10, 1)
    per_s = probe["times"][0] / 10.0
    dur = int(max(2, min(max_dur, budget_s / max(per_s, 1e-6))))
    return max(2, dur - dur % 2)


def cpu_baseline(name, budget_s=15.0):
    """The oracle on the host cores: single-threaded on a prefix sized to `budget_s`, and on every
    core (a process pool running the same oracle functions) on the longest prefix, up to the whole
    sequence, that the single-threaded rate predicts to fit in about the same time."""
    from synth import workload
    probe = run_oracle(name, 10, 1)
    per_s = probe["times"][0] / 10.0
    dur = int(max(2, min(360, budget_s / max(per_s, 1e-6))))
    dur -= dur % 2
    d = run_oracle(name, dur, 1)
    v1 = d["mm"] / d["times"][0]
    single = {"value": v1, "unit": UNIT, "cores": 1, "kind": "oracle",
              "sample": f"first {dur} s of the {name} sequence ({d['tokens']} tokens), same heads, query rows and "
                        f"schedule, single-threaded numpy fp64 oracle, {d['times'][0]:.1f} s"}
    workers = os.cpu_count() or 1
    if workers < 2:
        return {**single, **host_cpu()}
    full = workload(name).seqs[0].duration_s
    dur_p = int(max(2, min(full, 0.6 * budget_s * workers / max(per_s, 1e-6))))
    dur_p -= dur_p % 2
    try:
        p = run_oracle_pool(name, dur_p, workers)
    except Exception as exc:  # report, do not hide: the single-threaded number stands alone then
        return {**single, **host_cpu(), "parallel_error": str(exc)[-300:]}
    vp = p["mm"] / p["times"][0]
    what = "the whole sequence" if dur_p >= full else f"first {dur_p} s of the {name} sequence"
    return {"value": vp, "unit": UNIT, "cores": workers, "kind": "oracle", **host_cpu(),
            "sample": f"{what} ({p['tokens']} tokens), same heads, query rows and schedule; the numpy fp64 "
                      f"oracle's functions on a pool of {workers} single-threaded processes (scoring split over "
                      f"KV head groups and query-row chunks, row copies over planes, selection in the parent), "
                      f"{p['times'][0]:.1f} s after one warm-up pass",
            "single_thread": single}


def reference_arm(args, rank, world):
    if rank != 0:
        return
    per_step = min(10.0, 120.0 / max(1, args.steps + args.warmup))
    dur = cpu_sample_duration(args.workload, per_step)
    d = run_oracle(args.workload, dur, args.warmup + args.steps)
    times = d["times"][args.warmup:]
    t = sum(times)
    v = d["mm"] * len(times) / t
    sample = (f"first {dur} s of the {args.workload} sequence ({d['tokens']} tokens) per step, same heads, query "
              f"rows and 3-step schedule, single-threaded numpy fp64 oracle")
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * t / len(times), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": args.workload, "sample_seconds": dur},
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": sample, **host_cpu()},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


PRELLM_SNIPPET = r"""
import json, sys, time
sys.path.insert(0, {root!r})
import oracle
from synth.gen import normal_bf16_bits, TID_VIS_EMB, TID_AUD_EMB
F, tpf, na, dim = {F}, {tpf}, {na}, {dim}
vis = normal_bf16_bits({seed}, TID_VIS_EMB, 0, F * tpf * dim).reshape(F * tpf, dim)
aud = normal_bf16_bits({seed}, TID_AUD_EMB, 0, na * dim).reshape(na, dim)
t0 = time.perf_counter()
oracle.frame_alignment(vis, aud, F, tpf)
print(json.dumps(dict(seconds=time.perf_counter() - t0)))
"""


def prellm_shape(wl):
    """Frames, visual tokens per frame, audio tokens and feature size of the
    pre-LLM alignment of the workload's first sequence."""
    s = wl.seqs[0]
    return s.fps * s.duration_s, s.tpf, s.n_audio, wl.hidden


def prellm_cpu_baseline(wl, frames=24):
    F, tpf, na, dim = prellm_shape(wl)
    fs = min(F, frames)
    nas = max(fs, na * fs // F)
    env = dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1", MKL_NUM_THREADS="1")
    code = PRELLM_SNIPPET.format(root=ROOT, F=fs, tpf=tpf, na=nas, dim=dim, seed=wl.seed)
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env)
    if r.returncode != 0:
        raise RuntimeError(r.stderr[-2000:])
    sec = json.loads(r.stdout.strip().splitlines()[-1])["seconds"]
    return {"value": fs / sec, "unit": "frames/s", "cores": 1, "kind": "oracle", **host_cpu(),
            "sample": f"{fs} frames x {tpf} visual tokens, {nas} audio tokens, d={dim}; single-threaded numpy "
                      f"fp64 oracle (literal d x d products), {sec:.1f} s"}


def prellm_measure(ap, wl, steps, warmup, stream, dist, window=3):
    """Pre-LLM frame alignment (Sec. 3.1, Eq. cka and Eq. gate) of the
    workload's clip: pooled frame embeddings, windowed CKA and the gate, one
    apack_frame_alignment call per step.  The bf16 encoder tokens are read
    once and exceed L2, so no flush is needed between calls."""
    import torch
    from synth.gen import TID_VIS_EMB, TID_AUD_EMB
    from synth.device import fill_normal_bf16
    F, tpf, na, dim = prellm_shape(wl)
    vis = torch.empty(F * tpf, dim, dtype=torch.bfloat16, device="cuda")
    aud = torch.empty(na, dim, dtype=torch.bfloat16, device="cuda")
    fill_normal_bf16(vis, wl.seed, TID_VIS_EMB, stream=stream)
    fill_normal_bf16(aud, wl.seed, TID_AUD_EMB, stream=stream)
    ws = torch.empty(ap.apack_frame_alignment_workspace_size(F, dim), dtype=torch.uint8, device="cuda")
    c = torch.empty(F, dtype=torch.float32, device="cuda")
    sc = torch.empty_like(c)

    def call():
        ap.apack_frame_alignment(vis, aud, F, tpf, na, dim, c, sc, ws, window=window, stream=stream)

    for _ in range(max(3, warmup)):
        call()
    torch.cuda.synchronize()
    k = max(3, min(steps, 50))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    n0 = ap.apack_launch_count()
    e0.record(stream)
    for _ in range(k):
        call()
    e1.record(stream)
    torch.cuda.synchronize()
    launches = ap.apack_launch_count() - n0
    ms = max_over_ranks(e0.elapsed_time(e1) / k, dist, "cuda")
    token_bytes = (F * tpf + na) * dim * 2
    frame_bytes = 2 * F * dim * 4
    alg = token_bytes + frame_bytes
    achieved = alg / (ms / 1e3) / 1e9
    peak, peak_kind = measured_peaks()
    prof = profiled_traffic("prellm.cu", "prellm_traffic.json")
    traffic = int(prof["traffic_over_algorithmic"] * alg) if prof is not None else None
    del vis, aud, ws
    return {"metric": "frames aligned per second", "value": F / (ms / 1e3), "unit": "frames/s",
            "ms_per_clip": ms, "steps": k, "gpu_launches": int(launches),
            "config": {"workload": f"{wl.name} clip: {F} frames x {tpf} visual tokens, {na} audio tokens, d={dim}",
                       "window": window, "tau": 0.78, "beta": 0.90,
                       "l2": "inputs larger than L2 (%.2f GB of bf16 encoder tokens)" % (token_bytes / 1e9)},
            "roofline": {"bound": "hbm", "kernel": "apack_frame_alignment call (frame_pool_kernel + "
                                                   "frame_cka_gate_kernel)",
                         "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                         "traffic": traffic, "peak_source": peak_kind,
                         "algorithmic_bytes_per_launch": alg,
                         "note": "bf16 tokens read once + fp32 frame embeddings written once, over the whole call"}}


def final_levels_measure(ap, pp, nsteps, mm_per_iter, steps, warmup, stream, dist):
    """The same steps scheduled so that every layer's rows are written once, at the level that
    layer ends at (ProgressivePrune.run_from_host with the device inputs as its source): step i
    gathers layers [l_i, l_(i+1)) and the next step's scored keys from the step-0 input at the
    composed indices.  Same scores, selections and final caches as the per-step schedule (checked
    here against its last step's output); fewer bytes, because the per-step schedule compacts
    layers [l_i, L) at every step.  Reported beside the headline, not as it."""
    import torch
    lo = pp.layers[0]
    ref_k, ref_v = [x.clone() for x in pp.output_kv(nsteps - 1)]
    ref_h = pp.output_hidden(nsteps - 1).clone()

    def run():
        pp.run_from_host(pp.k_in, pp.v_in, pp.hidden_in, stream=stream)

    for _ in range(max(1, warmup)):
        run()
    torch.cuda.synchronize()
    k, v = pp.final_kv(nsteps - 1)
    same = (torch.equal(k.view(torch.int16), ref_k.view(torch.int16)) and
            torch.equal(v.view(torch.int16), ref_v.view(torch.int16)) and
            torch.equal(pp.output_hidden(nsteps - 1).view(torch.int16), ref_h.view(torch.int16)))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(steps):
        run()
    e1.record(stream)
    torch.cuda.synchronize()
    ms = max_over_ranks(e0.elapsed_time(e1) / steps, dist, "cuda")
    # the same calls captured once as a CUDA graph (stream capture of the library calls) and replayed
    graph_ms, graph_error = None, None
    try:
        graph = torch.cuda.CUDAGraph()
        cap = torch.cuda.Stream()
        cap.wait_stream(stream)
        with torch.cuda.graph(graph, stream=cap, capture_error_mode="thread_local"):
            pp.run_from_host(pp.k_in, pp.v_in, pp.hidden_in)
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            for _ in range(max(1, warmup)):
                graph.replay()
            torch.cuda.synchronize()
            g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            g0.record(stream)
            for _ in range(steps):
                graph.replay()
            g1.record(stream)
            torch.cuda.synchronize()
        graph_ms = max_over_ranks(g0.elapsed_time(g1) / steps, dist, "cuda")
        k, v = pp.final_kv(nsteps - 1)
        same = same and (torch.equal(k.view(torch.int16), ref_k.view(torch.int16)) and
                         torch.equal(v.view(torch.int16), ref_v.view(torch.int16)))
        del graph
    except Exception as exc:  # report, do not hide: the eager number stands alone then
        graph_error = str(exc)[-300:]
    moved = 0                         # read + write of every gathered row, 4 B index per kept row
    for i in range(nsteps):
        c, t = pp.fin_layers[i], pp.t_out[i]
        planes = 2 * c + (1 if i + 1 < nsteps else 0)
        moved += 2 * t * (planes * pp.row + (pp.H * 2 if i + 1 == nsteps else 0)) + 4 * t
    best = graph_ms if graph_ms is not None else ms
    return {"value": mm_per_iter / (best / 1e3), "unit": UNIT, "ms_per_step": best, "steps": steps,
            "eager_ms_per_step": ms, "graph_error": graph_error, "bytes_moved_per_iter": int(moved),
            "equal_to_per_step_schedule": bool(same),
            "how": "the library calls of ProgressivePrune.run_from_host captured once as a CUDA graph and replayed "
                   "(eager_ms_per_step: direct calls); every layer's K/V and the hidden states written once at their "
                   "final level from the step-0 input, the scored keys compacted per step; the per-step schedule "
                   "of the headline compacts layers [l_i, L) and the hidden states at every step"}


def link_rates(h_k, h_v, pp2, s_up, s_down, reps=3):
    """The host link's rate on this machine, measured beside the e2e run: pinned host -> device
    copies of up to 7 cache slabs alone, and the same copies while device -> host copies of as
    many bytes run on another stream (the e2e pipeline keeps both directions busy)."""
    import torch
    lo = 1 if h_k.shape[0] > 1 else 0
    n = min(lo + 7, h_k.shape[0])
    src, dst = h_k[lo:n], pp2.k_in[lo:n]
    back_src, back_dst = pp2.v_in[lo:n], h_v[lo:n]
    nbytes = src.numel() * src.element_size()

    def timed(both):
        best = None
        for _ in range(reps):
            torch.cuda.synchronize()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            if both:
                with torch.cuda.stream(s_down):
                    back_dst.copy_(back_src, non_blocking=True)
            with torch.cuda.stream(s_up):
                a.record(s_up)
                dst.copy_(src, non_blocking=True)
                b.record(s_up)
            torch.cuda.synchronize()
            ms = a.elapsed_time(b)
            best = ms if best is None else min(best, ms)
        return nbytes / (best / 1e3) / 1e9

    return {"h2d_gbs_alone": timed(False), "h2d_gbs_with_d2h": timed(True), "bytes": int(nbytes),
            "how": "pinned host -> device copy of %d cache slabs, best of %d, alone and beside a device -> host "
                   "copy of the same size" % (n - lo, reps)}


def scoring_roofline(wl, pp, cuq, score_ms_per_step, sm_mhz=None):
    """Useful tensor work of the scoring stage: one Q K^T over the multimodal keys per
    step and sequence (2 n_q Hq |S| D flop, summed over the sequences of the batch).  The two-pass softmax computes Q K^T twice and every
    logit also needs one exp2 per pass (the SFU is the second ceiling), so this
    fraction understates how busy the tensor pipe is: `frac_executed` counts both
    contractions, and `exp2_per_clk_per_sm` is the exp2 rate the stage sustained."""
    import numpy as np
    import torch
    nq = np.diff(np.asarray(cuq, np.int64))                   # query rows per sequence
    # |S| per sequence entering each step: the original counts, then the previous step's kept counts
    s_seq = [np.asarray(pp.na0, np.int64) + np.asarray(pp.nv0, np.int64)]
    s_seq += [np.asarray(c, np.int64).reshape(len(nq), 2).sum(axis=1) for c in pp.counts[:-1]]
    flops = [2.0 * wl.num_q_heads * wl.head_dim * float((nq * sq).sum()) for sq in s_seq]
    ms = float(np.sum(score_ms_per_step))
    achieved = sum(flops) / (ms / 1e3) / 1e12
    peak, kind = measured_tensor_peak()
    exp2 = 2 * sum(flops) / (2.0 * wl.head_dim)
    sms = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
    return {"bound": "tensor", "kernel": "score_rowstats_kernel + score_colsum_kernel (+ q_pack, merge, finalize)",
            "achieved": achieved, "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak, "traffic": None,
            "peak_source": kind, "useful_flops_per_iter": sum(flops),
            "executed_flops_per_iter": 2 * sum(flops), "frac_executed": 2 * achieved / peak,
            "logits_per_iter": sum(flops) / (2.0 * wl.head_dim), "exp2_per_iter": exp2,
            "exp2_per_clk_per_sm": (exp2 / (ms / 1e3) / sms / (sm_mhz * 1e6)) if sm_mhz else None,
            "note": "useful flops = one Q K^T per step over the multimodal keys; the stage runs two passes "
                    "(executed = both contractions) and one exp2 per logit in each"}


PAPER_WORKLOAD = "7b_10min_paper"


def paper_setting_measure(ap, steps, warmup, stream, dist, clocks=None):
    """The paper's own inner-LLM setting on the 10-minute 7B sequence (Sec. 3.2 with Table
    S-hparams: the last query token only, one top-k over all of S, a step at every layer from
    L_mid = 14 to 27 keeping 85 % of the current |S|): 14 prune steps per iteration, each
    scoring through the few-row path.  Timed as the headline is (the schedule captured once as
    a CUDA graph and replayed; stage events from direct apack_prune_schedule calls), with the
    HBM roofline of the few-row scoring (every step reads its layer's keys once) and of the
    compaction."""
    import numpy as np
    import torch
    from paper_2608_08794_gb300.schedule import ProgressivePrune, schedule_keep_counts
    from synth import workload
    from synth.device import fill_progressive_inputs
    wl = workload(PAPER_WORKLOAD)
    cu0, cuq = wl.cu_seqlens(), wl.cu_qlens()
    na = np.array([s.n_audio for s in wl.seqs], np.int32)
    nv = np.array([s.n_visual for s in wl.seqs], np.int32)
    mod_tmp = torch.from_numpy(wl.modality()).cuda()
    counts, mode = schedule_keep_counts(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, mod_tmp,
                                        len(wl.prune_layers), wl.ratios, wl.joint_step_keep)
    pp = ProgressivePrune(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, wl.num_layers, wl.hidden,
                          wl.prune_layers, counts, select_mode=mode)
    fill_progressive_inputs(pp, wl)
    nsteps = len(wl.prune_layers)
    mm = pp.mm_tokens_per_step()
    mm_per_iter = sum(mm)
    t_in = [wl.total_tokens] + list(pp.t_out[:-1])
    row = wl.num_kv_heads * wl.head_dim * 2
    for _ in range(max(1, warmup)):
        pp.run(stream=stream)
    torch.cuda.synchronize()
    ev = [[[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(nsteps)] for _ in range(steps)]
    for per_iter in ev:
        for per_step in per_iter:
            for e in per_step:
                e.record(stream)
    torch.cuda.synchronize()
    for k in range(steps):
        pp.run(events=ev[k], stream=stream)
    torch.cuda.synchronize()
    stage = np.zeros((nsteps, 3))
    for k in range(steps):
        for i in range(nsteps):
            for st in range(3):
                stage[i, st] += ev[k][i][st].elapsed_time(ev[k][i][st + 1])
    stage /= steps
    graph = pp.capture()
    for _ in range(max(1, warmup)):
        graph.launch(stream)
    torch.cuda.synchronize()
    g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    c0 = ap.apack_launch_count()
    if clocks:
        clocks.mark(True)
    g0.record(stream)
    for _ in range(steps):
        graph.launch(stream)
    g1.record(stream)
    torch.cuda.synchronize()
    if clocks:
        clocks.mark(False)
    launches = ap.apack_launch_count() - c0
    graph_ms = max_over_ranks(g0.elapsed_time(g1) / steps, dist, "cuda")
    graph.close()
    if ap.apack_device_error(pp.ws) != ap.APACK_OK:
        raise RuntimeError("the paper-setting schedule reported a device error")
    peak, peak_kind = measured_peaks()
    # few-row scoring: each step reads its layer's K rows (Hkv x 128 bf16 per token) and the modality byte
    # once and writes one fp32 score per token
    score_bytes = [t * (row + 1 + 4) for t in t_in]
    score_ms = stage[:, 0]
    score_gbs = sum(score_bytes) / (score_ms.sum() / 1e3) / 1e9
    comp_bytes = [2 * t * (2 * (wl.num_layers - l) * row + wl.hidden * 2) + 4 * t
                  for t, l in zip(pp.t_out, wl.prune_layers)]
    comp_ms = stage[:, 2]
    comp_gbs = sum(comp_bytes) / (comp_ms.sum() / 1e3) / 1e9
    out = {"workload": PAPER_WORKLOAD, "value": whole_job_value(mm_per_iter, 1 if dist is None else
                                                                  dist.get_world_size(), graph_ms),
           "unit": UNIT, "ms_per_step": graph_ms, "steps": steps, "gpu_launches": int(launches),
           "prune_layers": wl.prune_layers, "tokens_after_steps": pp.t_out, "mm_tokens_per_iter": mm_per_iter,
           "stages_ms_per_iter": {"score": float(score_ms.sum()), "select": float(stage[:, 1].sum()),
                                  "compact": float(comp_ms.sum())},
           "score_select_us_per_step": [float(1e3 * (a + b)) for a, b in zip(score_ms, stage[:, 1])],
           "roofline_scoring": {"bound": "hbm", "kernel": "few-row scoring (score_narrow_tc_kernel + merge + final)",
                                "achieved": score_gbs, "peak": peak, "unit": "GB/s", "frac": score_gbs / peak,
                                "traffic": None, "peak_source": peak_kind,
                                "algorithmic_bytes_per_iter": int(sum(score_bytes)),
                                "note": "per step and token: its K row (Hkv x 128 bf16) and modality byte read "
                                        "once, one fp32 score written"},
           "roofline_compaction": {"bound": "hbm", "kernel": "gather_tma_kernel", "achieved": comp_gbs,
                                   "peak": peak, "unit": "GB/s", "frac": comp_gbs / peak,
                                   "peak_source": peak_kind},
           "how": "the 14-step schedule captured once by apack_prune_schedule_graph and replayed; stage times "
                  "from direct apack_prune_schedule calls with stage events"}
    # the same 14 steps with every layer and the hidden states written once, at their final level
    out["schedule_final_levels"] = final_levels_measure(ap, pp, nsteps, mm_per_iter, steps, warmup, stream, dist)
    del pp
    torch.cuda.empty_cache()
    return out


def decode_measure(ap, wl, pp, steps, warmup, stream, dist):
    """Decode-step attention (one new token, Sec. 3.2 last sentence) over the
    layers compacted by the last prune step, on their uncompressed cache and on
    the compacted one: the decode-side effect of the schedule.  Each call is one
    layer; the calls rotate over the layers (more bytes than L2 holds)."""
    import torch
    from synth.gen import TID_Q
    from synth.device import fill_normal_bf16
    if wl.num_seqs != 1:
        return None
    last = len(pp.t_out) - 1
    l_last = wl.prune_layers[last]
    nl = wl.num_layers - l_last
    full_k = [pp.k_in[l_last - wl.prune_layers[0] + j] for j in range(nl)]
    full_v = [pp.v_in[l_last - wl.prune_layers[0] + j] for j in range(nl)]
    ck, cv = pp.output_kv(last)
    hq, hkv = wl.num_q_heads, wl.num_kv_heads
    q = torch.empty(1, hq, 128, dtype=torch.bfloat16, device="cuda")
    fill_normal_bf16(q, wl.seed, TID_Q + 999, stream=stream)
    out = torch.empty(1, hq, 128, dtype=torch.float32, device="cuda")
    res = {}
    for name, T, ks, vs in (("full", wl.total_tokens, full_k, full_v),
                            ("compacted", int(pp.t_out[last]), [ck[j] for j in range(nl)], [cv[j] for j in range(nl)])):
        cu = [0, T]
        ws = torch.zeros(max(256, ap.apack_decode_workspace_size(cu, hq, hkv)), dtype=torch.uint8, device="cuda")
        stride = hkv * 128 * 2

        def call(j):
            ap.apack_decode_attention(cu, q, ks[j], vs[j], stride, hq, hkv, out, ws, stream=stream)

        for j in range(max(3, warmup) * nl):
            call(j % nl)
        torch.cuda.synchronize()
        n = max(3, min(steps, 50)) * nl
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        c0 = ap.apack_launch_count()
        e0.record(stream)
        for j in range(n):
            call(j % nl)
        e1.record(stream)
        torch.cuda.synchronize()
        res[name] = (max_over_ranks(e0.elapsed_time(e1) / n, dist, "cuda"), T, ap.apack_launch_count() - c0, n)
    peak, peak_kind = measured_peaks()
    ms_full, T_full, launches, calls = res["full"]
    alg = T_full * hkv * 128 * 2 * 2 + hq * 128 * (2 + 4)
    achieved = alg / (ms_full / 1e3) / 1e9
    prof = profiled_traffic("decode_tc.cu", "decode_traffic.json") if hkv in (2, 4) and hq // hkv <= 8 else None
    traffic = int(prof["traffic_over_algorithmic"] * alg) if prof is not None else None
    kern = ("decode_tc_kernel + decode_combine_kernel" if hkv in (2, 4) and hq // hkv <= 8
            else "decode_chunk_kernel + decode_combine_kernel")
    return {"metric": "decode-step attention time per layer, uncompressed vs compacted cache",
            "layers": f"{l_last}..{wl.num_layers - 1}", "tokens": [T_full, res["compacted"][1]],
            "full_ms_per_layer": ms_full, "compacted_ms_per_layer": res["compacted"][0],
            "speedup": ms_full / res["compacted"][0], "calls_timed": calls,
            "gpu_launches_per_call": launches / calls,
            "roofline": {"bound": "hbm", "kernel": f"apack_decode_attention call on the uncompressed cache ({kern})",
                         "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                         "traffic": traffic, "peak_source": peak_kind, "algorithmic_bytes_per_launch": alg,
                         "note": "K and V of one layer read once, q read and out written once"}}


def decode_only(args):
    """Decode-step attention alone: one decode token of a single sequence over a synthetic
    cache of `--decode-tokens` keys (7B heads, 28 query / 4 KV), rotating over
    `--decode-layers` layers.  Prints one JSON line (time per layer, roofline)."""
    import torch
    import paper_2608_08794_gb300 as ap
    from synth.gen import TID_Q
    from synth.device import fill_normal_bf16
    hq, hkv, T, nl = 28, 4, args.decode_tokens, args.decode_layers
    stream = torch.cuda.current_stream()
    ks = [torch.empty(T, hkv * 128, dtype=torch.bfloat16, device="cuda") for _ in range(nl)]
    vs = [torch.empty(T, hkv * 128, dtype=torch.bfloat16, device="cuda") for _ in range(nl)]
    for j in range(nl):
        fill_normal_bf16(ks[j], 17, 2 * j, stream=stream)
        fill_normal_bf16(vs[j], 17, 2 * j + 1, stream=stream)
    q = torch.empty(1, hq, 128, dtype=torch.bfloat16, device="cuda")
    fill_normal_bf16(q, 17, TID_Q, stream=stream)
    out = torch.empty(1, hq, 128, dtype=torch.float32, device="cuda")
    cu = [0, T]
    ws = torch.zeros(max(256, ap.apack_decode_workspace_size(cu, hq, hkv)), dtype=torch.uint8, device="cuda")
    for j in range(args.warmup * nl):
        ap.apack_decode_attention(cu, q, ks[j % nl], vs[j % nl], hkv * 256, hq, hkv, out, ws, stream=stream)
    torch.cuda.synchronize()
    n = args.steps * nl
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for j in range(n):
        ap.apack_decode_attention(cu, q, ks[j % nl], vs[j % nl], hkv * 256, hq, hkv, out, ws, stream=stream)
    e1.record(stream)
    torch.cuda.synchronize()
    if ap.apack_device_error(ws) != ap.APACK_OK:
        raise RuntimeError("decode attention reported a device error")
    ms = e0.elapsed_time(e1) / n
    peak, peak_kind = measured_peaks()
    alg = T * hkv * 128 * 2 * 2 + hq * 128 * (2 + 4)
    achieved = alg / (ms / 1e3) / 1e9
    print(json.dumps({"metric": "decode-step attention time per layer", "value": ms, "unit": "ms",
                      "higher_is_better": False, "steps": args.steps, "warmup": args.warmup,
                      "config": {"workload": f"one sequence, {T} cached tokens, 28 query / 4 KV heads, "
                                             f"{nl} layers rotated", "dtype": "bf16"},
                      "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                                   "frac": achieved / peak, "peak_source": peak_kind,
                                   "algorithmic_bytes_per_launch": alg}}))


def compact_only(args):
    """The first prune step's compaction of the 10-minute 7B sequence alone: K and V of layers
    4..27 (48 planes of 135272 rows of 1024 B, 58772 kept; --compact-planes sets the plane count
    for a smaller profiling case), out of place (ping-pong buffers) and in place (src == dst),
    through apack_compact.  Prints one JSON line."""
    import numpy as np
    import torch
    import paper_2608_08794_gb300 as ap
    T, n_keep, planes, rb = 135272, 58772, args.compact_planes, 1024
    rng = np.random.default_rng(4)
    keep = torch.from_numpy(np.sort(rng.choice(T, n_keep, replace=False)).astype(np.int32)).cuda()
    src = torch.empty((planes, T, rb), dtype=torch.uint8, device="cuda")
    dst = torch.empty((planes, n_keep, rb), dtype=torch.uint8, device="cuda")
    ws = torch.zeros(1024, dtype=torch.uint8, device="cuda")
    alg = 2 * n_keep * rb * planes + 4 * n_keep
    peak, peak_kind = measured_peaks()
    out = {}
    for name, plane in (("out_of_place", ap.make_plane(src, dst, rb, planes, T * rb, n_keep * rb)),
                        ("in_place", ap.make_plane(src, src, rb, planes, T * rb, T * rb))):
        for _ in range(args.warmup):
            ap.apack_compact(keep, n_keep, [plane], ws=ws)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(args.steps):
            ap.apack_compact(keep, n_keep, [plane], ws=ws)
        e1.record()
        torch.cuda.synchronize()
        if ap.apack_device_error(ws) != ap.APACK_OK:
            raise RuntimeError("compaction reported a device error")
        ms = e0.elapsed_time(e1) / args.steps
        out[name] = {"ms": ms, "GB/s": alg / ms / 1e6, "frac": alg / ms / 1e6 / peak}
    print(json.dumps({"metric": "compaction time of the first 10-minute 7B prune step", "unit": "ms",
                      "higher_is_better": False, "steps": args.steps, "warmup": args.warmup,
                      "config": {"workload": f"{planes} planes x {T} rows of {rb} B, {n_keep} kept (random)",
                                 "l2": "inputs larger than L2 (%.1f GB)" % (planes * T * rb / 1e9)},
                      "peak": peak, "peak_source": peak_kind, "algorithmic_bytes": alg, **out}))


# ----------------------------------------------------------------------------- GPU leg

def main():
    args = parse()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        reference_arm(args, rank, world)
        return
    if args.part == "decode":
        decode_only(args)
        return
    if args.part == "compact":
        compact_only(args)
        return
    if args.part == "prellm":
        import torch
        import paper_2608_08794_gb300 as ap
        from synth import workload
        torch.cuda.set_device(local)
        print(json.dumps(prellm_measure(ap, workload(args.workload), args.steps, args.warmup,
                                        torch.cuda.current_stream(), None, window=args.window)))
        return

    import numpy as np
    import torch
    import paper_2608_08794_gb300 as ap
    from paper_2608_08794_gb300.schedule import ProgressivePrune, schedule_keep_counts
    from synth import workload
    from synth.device import fill_progressive_inputs

    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    def barrier():
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize()

    wl = workload(args.workload)
    # a batch of several sequences splits over the ranks by whole sequences (no data-path exchange:
    # each rank prunes and keeps its own sequences); a single sequence runs as one replica per rank
    sharded = world > 1 and wl.num_seqs >= world and not args.replicas
    if sharded:
        from paper_2608_08794_gb300.shard import plan_by_sequence
        from synth.configs import sequence_subset
        wl = sequence_subset(wl, plan_by_sequence(wl.cu_seqlens(), world)[rank])
    cu0, cuq = wl.cu_seqlens(), wl.cu_qlens()
    na = np.array([s.n_audio for s in wl.seqs], np.int32)
    nv = np.array([s.n_visual for s in wl.seqs], np.int32)
    mod_tmp = torch.from_numpy(wl.modality()).cuda()
    counts, mode = schedule_keep_counts(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, mod_tmp,
                                        len(wl.prune_layers), wl.ratios, wl.joint_step_keep)
    pp = ProgressivePrune(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, wl.num_layers, wl.hidden,
                          wl.prune_layers, counts, select_mode=mode)
    fill_progressive_inputs(pp, wl)
    mm_per_iter = sum(pp.mm_tokens_per_step())
    # units of the whole job per iteration: every rank's own sequences (split), or world replicas
    job_units = sum_over_ranks(mm_per_iter, dist, "cuda") if sharded else world * mm_per_iter
    nsteps = len(wl.prune_layers)
    stream = torch.cuda.current_stream()

    # algorithmic bytes of the compaction launch of each prune step
    row = wl.num_kv_heads * wl.head_dim * 2
    comp_bytes = [2 * t * (2 * (wl.num_layers - l) * row + wl.hidden * 2) + 4 * t
                  for t, l in zip(pp.t_out, wl.prune_layers)]

    def run_schedule(events=None):
        pp.run(events=events, stream=stream)     # the whole schedule: one apack_prune_schedule call

    for _ in range(args.warmup):
        run_schedule()
    torch.cuda.synchronize()

    # timed region: K iterations of the schedule; per step, events before scoring, after scoring,
    # after selection and after compaction, on the launching stream
    ev = [[[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(nsteps)]
          for _ in range(args.steps)]
    for per_iter in ev:       # torch creates events on first record; the C ABI records raw handles
        for per_step in per_iter:
            for e in per_step:
                e.record(stream)
    torch.cuda.synchronize()
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(local) if rank == 0 else None
    if clocks:
        clocks.start()
        time.sleep(0.3)
    launches0 = ap.apack_launch_count()
    barrier()
    if clocks:
        clocks.mark(True)
    t_start.record(stream)
    for k in range(args.steps):
        run_schedule(ev[k])
    t_end.record(stream)
    barrier()
    if clocks:
        clocks.mark(False)
    launches = ap.apack_launch_count() - launches0
    ms = max_over_ranks(t_start.elapsed_time(t_end), dist, "cuda")
    stage_ms = np.zeros((nsteps, 3))
    for k in range(args.steps):
        for i in range(nsteps):
            e = ev[k][i]
            for st in range(3):
                stage_ms[i, st] += e[st].elapsed_time(e[st + 1])
    stage_ms /= args.steps

    # the same schedule captured once into a CUDA graph (apack_prune_schedule_graph) and replayed:
    # the same launches with no per-kernel host launch between them
    graph = pp.capture()
    for _ in range(args.warmup):
        graph.launch(stream)
    g_start, g_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    g_launch0 = ap.apack_launch_count()
    barrier()
    if clocks:
        clocks.mark(True)
    g_start.record(stream)
    for _ in range(args.steps):
        graph.launch(stream)
    g_end.record(stream)
    barrier()
    if clocks:
        clocks.mark(False)
    g_launches = ap.apack_launch_count() - g_launch0
    graph_ms = max_over_ranks(g_start.elapsed_time(g_end) / args.steps, dist, "cuda")
    graph.close()
    final_levels = final_levels_measure(ap, pp, nsteps, mm_per_iter, args.steps, args.warmup, stream, dist)

    # end to end through the C ABI with host buffers: the caches of layers [l_0, L) and the hidden
    # states stay in pinned host memory.  Every iteration copies the scored layer's keys, the
    # queries and the modality to the device and runs the schedule from the host caches
    # (ProgressivePrune.host_step): each step scores and selects on the device and gathers over
    # the host link, at the composed indices, only the layers that end at its level (and the keys
    # the next step scores), so every layer's rows cross the link once.  The result (the last
    # step's layers, the hidden states, the indices) is read back.  Three device buffer sets let
    # iteration i+1's upload and first selection run while iteration i's gathers hold the link,
    # and iteration i-1's result is read back on a third stream (the link carries both
    # directions) without holding up iteration i+2's upload: with two sets, the gather queue
    # stood idle while one iteration's read-back, the next upload and its first selection ran.
    # Each step waits only for its own schedule's previous gather (not for gathers of the next
    # iteration queued meanwhile), so its scoring overlaps them; the next iteration's first
    # gather is queued before this iteration's last step, so the link never waits for a step's
    # scoring and selection.
    e2e_steps = args.e2e_steps or max(3, min(args.steps, 20))
    pp2, pp3 = (ProgressivePrune(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, wl.num_layers, wl.hidden,
                                 wl.prune_layers, counts, select_mode=mode) for _ in range(2))
    sets = [pp, pp2, pp3]
    h_k = torch.empty(pp.k_in.shape, dtype=pp.k_in.dtype, pin_memory=True)
    h_v = torch.empty_like(h_k, pin_memory=True)
    h_h = torch.empty(pp.hidden_in.shape, dtype=pp.hidden_in.dtype, pin_memory=True)
    h_m = torch.empty(pp.modality_in.shape, dtype=torch.uint8, pin_memory=True)
    h_q = [torch.empty(q.shape, dtype=q.dtype, pin_memory=True) for q in pp.q]
    h_k.copy_(pp.k_in); h_v.copy_(pp.v_in); h_h.copy_(pp.hidden_in); h_m.copy_(pp.modality_in)
    for a, b in zip(h_q, pp.q):
        a.copy_(b)
    last = nsteps - 1

    for p in sets:
        p._final_buffers()

    def host_outputs(p):
        ko, vo = p.final_kv(last)
        ho = p.output_hidden(last)
        return ([torch.empty(ko.shape, dtype=ko.dtype, pin_memory=True),
                 torch.empty(vo.shape, dtype=vo.dtype, pin_memory=True),
                 torch.empty(ho.shape, dtype=ho.dtype, pin_memory=True)] +
                [torch.empty(int(t), dtype=torch.int32, pin_memory=True) for t in p.t_out])

    h_out = [host_outputs(p) for p in sets]
    # bytes over the link per iteration: the copies (scored keys, modality, queries) and the rows
    # the gathers read from host memory (step i: the V of its layers, their K but for its scored
    # layer's after step 0, the next step's scored keys; the last step also the hidden states)
    h2d = h_k[0].numel() * h_k.element_size() + h_m.numel() + sum(x.numel() * x.element_size() for x in h_q)
    for i in range(nsteps):
        c = pp.fin_layers[i]
        planes = 2 * c - (1 if i > 0 else 0) + (1 if i + 1 < nsteps else 0)
        h2d += pp.t_out[i] * (planes * pp.row + (pp.H * 2 if i + 1 == nsteps else 0))
    d2h = sum(x.numel() * x.element_size() for x in h_out[0])
    # the device work of the e2e pipeline runs on a stream of the highest priority, so that its
    # kernels take SMs as soon as CTAs of the link-bound gather (default priority) retire
    stream_dev = stream
    stream = torch.cuda.Stream(priority=torch.cuda.Stream.priority_range()[1])
    stream.wait_stream(stream_dev)
    s_up, s_gather, s_down = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    ev_up = [torch.cuda.Event() for _ in sets]
    ev_comp = [torch.cuda.Event() for _ in sets]
    ev_down = [torch.cuda.Event() for _ in sets]
    for e in ev_down:
        e.record(stream)

    def front(j):
        """Upload, score, select and start the host-source compaction of iteration j."""
        b = j % len(sets)
        p = sets[b]
        with torch.cuda.stream(s_up):          # upload once the set's last result was read back
            s_up.wait_event(ev_down[b])
            p.k_in[0].copy_(h_k[0], non_blocking=True)      # the scored layer's keys
            p.modality_in.copy_(h_m, non_blocking=True)
            for a, qh in zip(p.q, h_q):
                a.copy_(qh, non_blocking=True)
            ev_up[b].record(s_up)
        stream.wait_event(ev_up[b])
        p.host_step(0, h_k, h_v, h_h, stream=stream, gather_stream=s_gather)

    def middle(j):
        """Steps 1 .. n-2 of iteration j."""
        p = sets[j % len(sets)]
        for i in range(1, nsteps - 1):
            p.host_step(i, h_k, h_v, h_h, stream=stream, gather_stream=s_gather)

    def back(j):
        """The last step and the read-back of iteration j."""
        b = j % len(sets)
        p = sets[b]
        if nsteps > 1:
            p.host_step(nsteps - 1, h_k, h_v, h_h, stream=stream, gather_stream=s_gather)
        ev_comp[b].record(stream)
        with torch.cuda.stream(s_down):
            s_down.wait_event(ev_comp[b])
            ko, vo = p.final_kv(last)
            o = h_out[b]
            o[0].copy_(ko, non_blocking=True); o[1].copy_(vo, non_blocking=True)
            o[2].copy_(p.output_hidden(last), non_blocking=True)
            for i, t in enumerate(p.t_out):
                o[3 + i].copy_(p.keep_idx[i][:t], non_blocking=True)
            ev_down[b].record(s_down)

    def e2e_run(n):
        # software pipeline: iteration j+1's upload, scoring, selection and first gather are
        # queued before iteration j's last step, so that the link carries that gather while the
        # last step scores and selects, and the last step's scoring runs during it
        front(0)
        for j in range(n):
            middle(j)
            if j + 1 < n:
                front(j + 1)
            back(j)

    e2e_run(len(sets))
    torch.cuda.synchronize()
    barrier()
    if clocks:
        clocks.mark(True)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    s_up.wait_stream(stream)
    s_gather.wait_stream(stream)
    e2e_run(e2e_steps)
    stream.wait_stream(s_down)
    e1.record(stream)
    barrier()
    if clocks:
        clocks.mark(False)
    e2e_ms = max_over_ranks(e0.elapsed_time(e1) / e2e_steps, dist, "cuda")
    link = link_rates(h_k, h_v, pp2, s_up, s_down)
    stream_dev.wait_stream(stream)
    stream = stream_dev
    del pp2, pp3, sets

    # the paper's own setting (last query token, joint top-k, 14 steps), when the headline is the
    # workloads' schedule
    paper = None
    if args.workload != PAPER_WORKLOAD and not args.no_paper_setting:
        paper = paper_setting_measure(ap, args.steps, args.warmup, stream, dist, clocks)
    # the pre-LLM stage of the same clip, timed on its own after the prune steps
    prellm = prellm_measure(ap, wl, args.steps, args.warmup, stream, dist)
    # decode-step attention over the last step's layers, before and after pruning
    decode = decode_measure(ap, wl, pp, args.steps, args.warmup, stream, dist)
    if clocks:
        clocks.stop()

    if rank == 0:
        eager_ms = ms / args.steps
        per_step_ms = graph_ms                     # the headline: the captured schedule, replayed
        value = job_units / (per_step_ms / 1e3)
        peak, peak_kind = measured_peaks()
        comp_ms = stage_ms[:, 2]
        achieved = sum(comp_bytes) / (comp_ms.sum() / 1e3) / 1e9
        prof = profiled_traffic(GATHER_SOURCES)
        traffic = None
        if prof is not None:   # ncu DRAM bytes of a captured launch, scaled to each launch by rows moved
            traffic = [int(prof["traffic_over_algorithmic"] * b) for b in comp_bytes]
        score_ms, select_ms = stage_ms[:, 0].sum(), stage_ms[:, 1].sum()
        clock_summary = clocks.summary() if clocks else {}
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": per_step_ms, "higher_is_better": True, "scaling": "strong" if sharded else "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": args.workload, "tokens": wl.total_tokens, "mm_tokens": wl.total_mm,
                       "query_rows": int(cuq[-1]), "heads": f"{wl.num_q_heads}q/{wl.num_kv_heads}kv",
                       "hidden": wl.hidden, "num_layers": wl.num_layers, "prune_layers": wl.prune_layers,
                       "tokens_after_steps": pp.t_out, "mm_tokens_per_iter": mm_per_iter,
                       "l2": "inputs larger than L2 (K/V of the compacted layers: %.1f GB)" %
                             (2 * pp.k_in.numel() * 2 / 1e9),
                       "parallelism": (f"{world} ranks, the batch's sequences split by tokens (rank 0's share "
                                       "shown above)" if sharded else
                                       f"{world} independent replicas" if world > 1 else "1 GPU")},
            "gpu_launches": int(g_launches),
            "roofline": {"bound": "hbm", "kernel": "gather_tma_kernel (compaction)", "achieved": achieved,
                         "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                         "traffic": traffic, "peak_source": peak_kind,
                         "algorithmic_bytes_per_launch": comp_bytes,
                         "avg_launch_ms": [float(x) for x in comp_ms]},
            "roofline_scoring": scoring_roofline(wl, pp, cuq, stage_ms[:, 0], clock_summary.get("sm_mhz")),
            "stages_ms_per_iter": {"score": float(score_ms), "select": float(select_ms),
                                   "compact": float(comp_ms.sum())},
            "launch": "the schedule captured once by apack_prune_schedule_graph and replayed every iteration "
                      "(apack_graph_launch)",
            "eager": {"value": job_units / (eager_ms / 1e3), "unit": UNIT,
                      "ms_per_step": eager_ms, "gpu_launches": int(launches),
                      "how": "one apack_prune_schedule call per iteration with stage events; stages_ms_per_iter "
                             "and the compaction roofline come from this run"},
            "schedule_final_levels": dict(final_levels, value=job_units / (final_levels["ms_per_step"] / 1e3)),
            "e2e": {"value": job_units / (e2e_ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": int(h2d),
                    "d2h_bytes_per_step": int(d2h), "ms_per_step": e2e_ms, "steps": e2e_steps,
                    "pipeline": "caches and hidden states in pinned host memory; per iteration the scored layer's "
                                "keys, the queries and the modality are copied; every step scores and selects on the "
                                "device and gathers over the host link (its own stream), at the composed indices, "
                                "the layers that end at its level plus the keys the next step scores (the last step "
                                "also the hidden states), so each layer's rows and the hidden states cross the link "
                                "once; the result is every layer's final cache on the "
                                "device, of which the last step's layers, the hidden states and the indices are read "
                                "back; three device buffer sets let the next iteration's upload and first selection "
                                "and the previous read-back run while the current gathers hold the link",
                    "h2d_note": "h2d_bytes_per_step counts the copies and the kept rows read from host memory",
                    "h2d_gbs": h2d / (e2e_ms / 1e3) / 1e9, "link": link,
                    "frac_of_link": (h2d / (e2e_ms / 1e3) / 1e9) / link["h2d_gbs_alone"]},
            "clocks": clock_summary or None,
            "context": schedule_context(wl, pp),
        }
        line["paper_setting"] = paper
        line["prellm_alignment"] = prellm
        line["decode_attention"] = decode
        if world == 1 and not args.no_cpu_baseline:
            try:
                line["cpu_baseline"] = cpu_baseline(args.workload)
            except Exception as exc:  # report, do not hide
                line["cpu_baseline"] = {"value": None, "error": str(exc)[-300:]}
            try:
                prellm["cpu_baseline"] = prellm_cpu_baseline(wl)
            except Exception as exc:
                prellm["cpu_baseline"] = {"value": None, "error": str(exc)[-300:]}
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
