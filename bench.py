"""Benchmark of one rollout-collection step (Algorithm 1 with batched bf16 decode) on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload 1.5b|3b|oversampled|tiny]
    python bench.py --impl reference ...      # the CPU oracle as the reference arm

A step is one sara_collect_step over a fresh synthetic prompt stream of the named workload:
probe, decide, refill and decode every issued rollout until the target or the budget is
reached.  Every step, warm-up and timed alike, goes through the public call with the
step's inputs in pinned host memory and its results copied back to pinned host memory, so
the timed steps are the end-to-end ones:

  * `value` = rollout tokens generated per second of the steps' device time with inputs
    already resident in HBM (the library's CUDA events after the input copies and before the
    output copies of each call), whole job over all ranks;
  * `e2e` = the same metric over the whole timed region (CUDA events on the handle's stream
    around the K calls, host<->device copies included).

N > 1 runs one replica per GPU on its own shard of the prompt stream (seed offset by rank, no
collective on the data path); only the final counters are reduced.  Rank 0 prints one JSON
line.  Data are synthetic (random-init weights, seeded rewards and lengths).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import platform
import subprocess
import sys
import tempfile
import time
from dataclasses import replace

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

HERE_PEAKS = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_HBM_GBS = 6800.0
CPU_SLICE_STEPS = 8        # decode steps of the oracle's teacher-forced slice
CPU_ONE_THREAD_LAYERS = 2  # layers timed on one thread (scaled to the whole model)


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="mine", choices=["mine", "reference"])
    ap.add_argument("--workload", default="1.5b", choices=sorted(synth.WORKLOADS))
    ap.add_argument("--schedule", type=int, default=0, choices=[0, 1, 2],
                    help="0: Algorithm 1's synchronised rounds (the paper's method, the default); 1 / 2: the "
                         "asynchronous per-prompt schedule without / with the budget reserve")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--kernel-profile", type=int, default=None, metavar="KERNEL",
                    help="profiling mode for ncu: launch one decode kernel (sara_profile ids; 0 = whole "
                         "eager decode step) on a reduced-capacity handle of the workload's shapes")
    ap.add_argument("--rows", type=int, default=25, help="live rows in --kernel-profile mode")
    ap.add_argument("--iters", type=int, default=5, help="launches in --kernel-profile mode")
    ap.add_argument("--points", default=None, metavar="RxC,...",
                    help="--kernel-profile mode: time the decode-step kernel (1) and the whole decode step (0) "
                         "at each rows x context point with one handle, e.g. 1x384,26x758,128x300 "
                         "(the comparison points of the design notes' A/B tables)")
    ap.add_argument("--ctx", type=int, default=None, help="context length in --kernel-profile mode "
                    "(default: prompt length + 128)")
    ap.add_argument("--controller", action="store_true",
                    help="time the on-device controller alone (controller-only handles) over the sweep grid "
                         "k x n0 x tau at P = 65,536: microseconds per round and decisions per second")
    ap.add_argument("--cpu-slice", action="store_true", help=argparse.SUPPRESS)  # child of the CPU baseline
    ap.add_argument("--slice-layers", type=int, default=None, help=argparse.SUPPRESS)
    return ap.parse_args()


# --------------------------------------------------------------------------------- helpers
def peaks():
    try:
        with open(HERE_PEAKS) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def cpu_model() -> str:
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    return platform.machine()


class ClockSampler:
    """nvidia-smi SM clocks and throttle reasons sampled every 200 ms during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu: int):
        self.gpu = gpu
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        rows = []
        try:
            for line in open(self.path):
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        except Exception:
            pass
        finally:
            try:
                os.unlink(self.path)
            except Exception:
                pass
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}

        def num(x):
            try:
                return float(x)
            except ValueError:
                return float("nan")
        sm = [num(r[1]) for r in rows]
        mx = [num(r[2]) for r in rows]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower().startswith("active")})
        loaded = [s for s in sm if not math.isnan(s)]
        return {"sm_mhz": float(np.median(loaded)) if loaded else None,
                "sm_max_mhz": float(np.nanmax(mx)) if mx else None, "reasons": reasons,
                "samples": len(rows)}


# ------------------------------------------------------------------------ algorithmic bytes
def weight_bytes_per_step(m: synth.ModelShape) -> int:
    """Every layer's weights and norms, the final norm and lm_head: read once per decode step."""
    return m.layers * (m.layer_weight_bytes() + 4 * m.d_model) + 2 * m.vocab * m.d_model + 2 * m.d_model


def decode_token_bytes(m: synth.ModelShape, Lp: int, lens: np.ndarray) -> float:
    """Per-token part of the decode bytes of rollouts with generated lengths `lens`: the K/V of
    the whole context read (contexts Lp, Lp+1, .., Lp+L-1), the new K/V written, the embedding
    rows.  The weight part (weight_bytes_per_step per decode step) is added by the caller."""
    kvtok = m.kv_bytes_per_token()
    L = lens.astype(np.float64)
    ctx_sum = (L * Lp + L * (L - 1) / 2).sum()
    return ctx_sum * kvtok + L.sum() * kvtok + L.sum() * m.d_model * 2


def step_algorithmic_bytes(m: synth.ModelShape, rows: int, ctx: int) -> float:
    """Bytes one decode step over `rows` rows at context `ctx` must move."""
    kvtok = m.kv_bytes_per_token()
    return weight_bytes_per_step(m) + rows * (ctx - 1) * kvtok + rows * kvtok + rows * m.d_model * 2


def executed_lengths(si, n: np.ndarray) -> np.ndarray:
    return np.concatenate([si.lengths[q, :int(n[q])] for q in range(len(n)) if n[q] > 0] or [np.zeros(0)])


# --------------------------------------------------------------------------------- CPU arm
def _slice_tokens(w: synth.Workload):
    """Inputs of the oracle's teacher-forced slice: the first prompt of round 0 and
    CPU_SLICE_STEPS forced generated tokens (the oracle's cost does not depend on their values)."""
    si = synth.step_inputs(w)
    return si, si.tokens[0], si.tokens[1, :CPU_SLICE_STEPS]


def time_slice(workload: str, layers: int | None = None, repeat: int = 1) -> list[float]:
    """Seconds of O2's teacher-forced slice (the first CPU_SLICE_STEPS decode steps of one
    round-0 rollout, by the oracle's full recompute over the prompt) on the model's first
    `layers` layers (all by default), `repeat` times, with this process's BLAS threads."""
    from oracle import decode as o2
    w = synth.WORKLOADS[workload]
    m = w.model
    L = m.layers if layers is None else layers
    weights = synth.global_weights(m, w.weight_seed)
    weights["layers"] = [synth.layer_weights(m, l, w.weight_seed) for l in range(L)]
    W = o2.Weights(replace(m, layers=L), weights)
    _, prompt, forced = _slice_tokens(w)
    out = []
    for _ in range(repeat):
        t0 = time.perf_counter()
        o2.teacher_forced_logits(W, prompt, forced)
        out.append(time.perf_counter() - t0)
    return out


def cpu_slice_child(args):
    """Child process of the CPU baseline (BLAS threads set by the parent's environment)."""
    print(json.dumps({"seconds": time_slice(args.workload, args.slice_layers)[0]}))


def _run_slice(workload: str, one_thread: bool, layers: int | None) -> float:
    env = dict(os.environ)
    if one_thread:  # BLAS on one thread (the input generator keeps its OpenMP threads)
        for k in ("OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS", "BLIS_NUM_THREADS"):
            env[k] = "1"
    cmd = [sys.executable, os.path.abspath(__file__), "--cpu-slice", "--workload", workload]
    if layers is not None:
        cmd += ["--slice-layers", str(layers)]
    r = subprocess.run(cmd, capture_output=True, text=True, env=env, timeout=900)
    if r.returncode != 0:
        raise RuntimeError(f"oracle slice failed: {r.stderr[-2000:]}")
    return float(json.loads(r.stdout.strip().splitlines()[-1])["seconds"])


def cpu_baseline(workload: str) -> dict:
    """The oracle as it stands, timed on this host's cores on a bounded sample of the workload:
    O1 (plain C, one thread) over the whole step's schedule, and O2 (float64 numpy) on the
    teacher-forced slice of one round-0 rollout, on all host threads (the whole model) and on
    one thread (CPU_ONE_THREAD_LAYERS layers, scaled to the whole model; the lm_head part is
    timed alone and not scaled).  value = O2 decode tokens per second on all threads."""
    from oracle import controller as oc
    w = synth.WORKLOADS[workload]
    m = w.model
    si, _, _ = _slice_tokens(w)
    t0 = time.perf_counter()
    oc.collect_workload(w, si)
    o1_s = time.perf_counter() - t0
    t_all = _run_slice(workload, False, None)
    t_head = _run_slice(workload, True, 0)
    t_part = _run_slice(workload, True, CPU_ONE_THREAD_LAYERS)
    t_one = t_head + (t_part - t_head) * m.layers / CPU_ONE_THREAD_LAYERS
    ncpu = os.cpu_count()
    try:
        avail = len(os.sched_getaffinity(0))
    except Exception:
        avail = ncpu
    return {
        "value": CPU_SLICE_STEPS / t_all, "unit": "rollout tokens/s", "cores": avail, "kind": "oracle",
        "sample": (f"O2 float64 teacher-forced slice: the first {CPU_SLICE_STEPS} decode steps of one of round 0's "
                   f"{w.target_B * w.n0} rollouts (the oracle's full recompute over the {w.prompt_len}-token prompt "
                   f"+ {CPU_SLICE_STEPS - 1} tokens), extrapolated to tokens/s = {CPU_SLICE_STEPS} / time; "
                   f"BLAS on all {avail} host threads; plus O1 over the whole step's schedule"),
        "o2_all_threads_s": round(t_all, 3), "o2_all_threads_tokens_per_s": CPU_SLICE_STEPS / t_all,
        "o2_one_thread_s": round(t_one, 3), "o2_one_thread_tokens_per_s": CPU_SLICE_STEPS / t_one,
        "o2_one_thread_note": (f"{CPU_ONE_THREAD_LAYERS} of {m.layers} layers timed on one thread and scaled; "
                               f"lm_head part timed alone ({t_head:.2f} s)"),
        "o1_whole_step_s": round(o1_s, 4), "o1_threads": 1,
        "os_cpu_count": ncpu, "cpu_model": cpu_model(), "machine": platform.machine(),
    }


# --------------------------------------------------------------------------------- GPU arm
def run_mine(args):
    import torch
    import torch.distributed as dist

    import paper_2607_26253_gb300 as pkg
    from paper_2607_26253_gb300 import replicas

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    t_start = time.time()
    # the CPU baseline first (rank 0 at N = 1 only): bounded, in child processes, before any
    # CUDA call of this process
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(args.workload)
    if world > 1:
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    w0 = synth.WORKLOADS[args.workload]
    m = w0.model
    w = w0.with_seed_offset(replicas.seed_offset(rank))  # each replica its own prompt-stream shard
    weights = synth.model_weights(m, w.weight_seed)
    cfg = pkg.model_cfg(m, max_prompts=w.n_prompts, max_active=w.target_B, max_seqs=w.target_B * w.n0,
                        max_prompt_len=w.prompt_len, max_gen_len=w.lengths.max_len, max_k=w.k)
    stream = torch.cuda.current_stream(dev)
    h = pkg.Handle(cfg, weights, stream=stream)
    del weights

    def pinned(a):
        t = torch.empty(a.shape, dtype=torch.from_numpy(a[:0]).dtype, pin_memory=True)
        t.numpy()[...] = a
        return t.numpy()

    # one synthetic batch per step: a fresh prompt stream (seeds shifted by the step index),
    # staged in pinned host memory; results land in pinned host buffers
    batches = []
    for i in range(args.warmup + args.steps):
        wi = w.with_seed_offset(7 * (i + 1))
        si = synth.step_inputs(wi)
        batches.append((wi, si, pinned(si.thresholds), pinned(si.lengths), pinned(si.tokens)))
    P = w.n_prompts
    outs_host = {"status": pinned(np.zeros(P, np.uint8)), "n": pinned(np.zeros(P, np.uint8)),
                 "s": pinned(np.zeros(P, np.uint8)), "decided_round": pinned(np.zeros(P, np.int16)),
                 "tokens": pinned(np.zeros((P, w.k, cfg.max_gen_len), np.int32))}

    def step(b):
        wi, _, thr, lens, toks = b
        return h.collect_step(thresholds=thr, lengths=lens, tokens=toks, N=wi.budget_N, k=wi.k, n0=wi.n0,
                              tau=wi.tau, target_B=wi.target_B, reward_seed=wi.reward_seed,
                              sample_seed=wi.sample_seed, commit_min=wi.commit_floor, prior=wi.prior,
                              want_tokens=True, outputs=outs_host, schedule=args.schedule)

    warm_s = []
    for i in range(args.warmup):
        t0 = time.time()
        step(batches[i])
        warm_s.append(time.time() - t0)
    if warm_s:
        print(f"[bench] {args.warmup} warm-up steps, {np.mean(warm_s):.1f} s each; {args.steps} timed steps "
              f"projected {np.mean(warm_s) * args.steps:.0f} s (setup {t_start and time.time() - t_start:.0f} s "
              f"so far)", file=sys.stderr, flush=True)

    # ------------------------------------------------------------------ timed region
    outs, n_executed = [], []
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    with ClockSampler(local) as clk:
        e0.record(stream)
        for i in range(args.warmup, args.warmup + args.steps):
            o = step(batches[i])
            outs.append(o)
            n_executed.append(o.n.copy())
        e1.record(stream)
        torch.cuda.synchronize(dev)
    if world > 1:
        dist.barrier()
    e2e_ms = e0.elapsed_time(e1)
    clocks = clk.summary()

    dev_ms = sum(o.device_ms for o in outs)
    k_ms_live = sum(o.decode_kernel_ms for o in outs)
    tok = sum(o.counters["gen_tokens"] for o in outs)
    groups = sum(o.counters["committed"] for o in outs)
    rollouts = sum(o.counters["rollouts"] for o in outs)
    dsteps = sum(o.counters["decode_steps"] for o in outs)
    rounds = sum(o.counters["rounds"] for o in outs)
    dec_bytes = 0.0
    for (wi, si, *_), o, n in zip(batches[args.warmup:], outs, n_executed):
        dec_bytes += decode_token_bytes(m, wi.prompt_len, executed_lengths(si, n)) + \
            o.counters["decode_steps"] * weight_bytes_per_step(m)
    b0 = batches[0]
    h2d = b0[2].nbytes + b0[3].nbytes + b0[4].nbytes
    d2h = sum(a.nbytes for a in outs_host.values())

    # cross-check of the dominant kernel with CUDA events around a captured graph of its
    # launches, at the timed steps' mean live rows and the median mid-rollout context
    mean_rows = max(1, int(round(tok / max(dsteps, 1))))
    mid_ctx = w.prompt_len + int(np.median(b0[1].lengths)) // 2
    k_ms = h.profile(1, mean_rows, mid_ctx, iters=20)
    k_bytes = step_algorithmic_bytes(m, mean_rows, mid_ctx)
    h.close()

    # ------------------------------------------------------------------ reduce over ranks
    if world > 1:  # the only collective: job totals (sum) over the slowest rank's time (max)
        dev_ms, e2e_ms, k_ms_live = replicas.reduce_max([dev_ms, e2e_ms, k_ms_live], device=dev)
        tok, groups, rollouts, dec_bytes = replicas.reduce_sum([tok, groups, rollouts, dec_bytes], device=dev)
    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    peak, peak_kind = peaks()
    achieved = dec_bytes / world / (k_ms_live * 1e-3) / 1e9  # per GPU: each replica's own kernel
    achieved_x = k_bytes / (k_ms * 1e-3) / 1e9
    tr = read_traffic(args.workload)
    per_launch = dec_bytes / world / max(dsteps, 1)
    traffic = None if tr is None else tr[0] * per_launch / tr[1]
    line = {
        "metric": "rollout tokens/sec (also effective groups/sec and decode HBM GB/s)",
        "value": tok / (dev_ms * 1e-3),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": dev_ms / args.steps,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (random-init weights N(0,0.02), seeded prompts, rewards and lengths)",
        "config": {"workload": w0.name + ("" if args.schedule == 0 else
                                          f" [asynchronous schedule{' + reserve' if args.schedule == 2 else ''}]"),
                   "global_batch": w0.target_B * world, "seq_len": w0.prompt_len,
                   "parallelism": f"replicas x{world} (prompt-stream shards)",
                   "l2": "inputs larger than L2 (3+ GB of weights streamed per decode step)"},
        "effective_groups_per_s": groups / (dev_ms * 1e-3),
        "rollouts_per_s": rollouts / (dev_ms * 1e-3),
        "decode_hbm_gbs": dec_bytes / world / (dev_ms * 1e-3) / 1e9,
        "decode_hbm_frac": dec_bytes / world / (dev_ms * 1e-3) / 1e9 / peak,
        "decode_steps_per_step": dsteps / world / args.steps,
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic,
                     "kernel": "decode_step_kernel (one launch = one whole decode forward over the live rows)",
                     "how": ("algorithmic bytes of every decode step of the timed steps (weights once + K/V of "
                             "every context position + K/V appends + embedding rows) / summed launch durations "
                             "(device clock per launch: earliest CTA start to latest CTA end)"),
                     "launches": dsteps // world, "bytes_per_launch_mean": per_launch,
                     "traffic_note": None if tr is None else "ncu DRAM bytes of one captured launch, scaled by algorithmic bytes",
                     "events_check": {"rows": mean_rows, "ctx": mid_ctx, "ms_per_launch": k_ms,
                                      "achieved": achieved_x, "frac": achieved_x / peak,
                                      "how": "CUDA events around 20 graph-captured launches at these rows and context"},
                     "peak_kind": f"{peak_kind} burst copy"},
        "e2e": {"value": tok / (e2e_ms * 1e-3), "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h,
                "how": "CUDA events around the K calls (pinned host inputs in, pinned host results out)"},
        "cpu_baseline": cpu,
        "gpu_launches": None,
        "clocks": clocks,
        "wall_s": round(time.time() - t_start, 1),
    }
    # kernels launched: per decode step the controller, the decode-step kernel and the
    # sampling/bookkeeping kernel; per round start (or, asynchronous, per decision event) at most
    # the prefill (embedding + 5 per layer but the last layer's 4) and the KV set-up; per call
    # the init kernel
    line["gpu_launches"] = int(3 * dsteps + rounds * (1 + 5 * m.layers - 4 + 1) + args.steps * world)
    line["committed_per_step"] = groups / world / args.steps
    line["kv_blocks_peak"] = max(o.kv_blocks_peak for o in outs)
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def read_traffic(workload: str):
    """(DRAM bytes, algorithmic bytes) of one launch of the dominant kernel from the committed
    ncu summary of the workload's model shape, or None."""
    shape = {"1.5b": "1p5b", "oversampled": "1p5b", "3b": "3b"}.get(workload)
    for kind in ("ncu", "dram"):
        path = os.path.join(ROOT, "profiles", f"decode_step_{shape}_{kind}.md")
        got = {}
        try:
            for line in open(path):
                for key in ("traffic_bytes_per_launch:", "algorithmic_bytes_per_launch:"):
                    if line.startswith(key):
                        got[key] = float(line.split(":", 1)[1].split()[0])
        except OSError:
            continue
        if len(got) == 2:
            return got["traffic_bytes_per_launch:"], got["algorithmic_bytes_per_launch:"]
    return None


# --------------------------------------------------------------------------------- ncu mode
def run_kernel_profile(args):
    """Small-footprint run of the real decode kernels for ncu captures: the workload's model
    shapes with 32 rollout slots of 512 generated positions (a few GB on the device)."""
    import torch

    import paper_2607_26253_gb300 as pkg
    torch.cuda.set_device(0)
    w = synth.WORKLOADS[args.workload]
    m = w.model
    weights = synth.model_weights(m, w.weight_seed)
    ctx = args.ctx if args.ctx is not None else w.prompt_len + 128
    gen = max(512, ctx - w.prompt_len + 2 * args.iters + 8)
    cfg = pkg.model_cfg(m, max_prompts=w.n_prompts, max_active=max(16, args.rows), max_seqs=max(32, args.rows),
                        max_prompt_len=w.prompt_len, max_gen_len=gen, max_k=w.k)
    if args.points:
        pts = [tuple(int(v) for v in p.split("x")) for p in args.points.split(",")]
        rmax, cmax = max(r for r, _ in pts), max(c for _, c in pts)
        cfg = pkg.model_cfg(m, max_prompts=w.n_prompts, max_active=max(16, rmax), max_seqs=max(32, rmax),
                            max_prompt_len=w.prompt_len, max_gen_len=max(512, cmax - w.prompt_len + 2 * args.iters + 8),
                            max_k=w.k)
        with pkg.Handle(cfg, weights, stream=torch.cuda.current_stream()) as h:
            for rows, c in pts:
                k1 = h.profile(1, rows, c, iters=args.iters)
                k0 = h.profile(0, rows, c, iters=args.iters)
                print(json.dumps({"rows": rows, "ctx": c, "kernel_ms": round(k1, 4), "step_ms": round(k0, 4)}), flush=True)
        return
    with pkg.Handle(cfg, weights, stream=torch.cuda.current_stream()) as h:
        ms = h.profile(args.kernel_profile, args.rows, ctx, iters=args.iters)
    print(json.dumps({"kernel": args.kernel_profile, "rows": args.rows, "ctx": ctx, "ms_per_launch": ms}))


# --------------------------------------------------------------------------------- controller
def run_controller(args):
    """The SARA controller kernel alone (Algorithm 1's rounds without decode) on the 63-point
    sweep grid at P = 65,536, B = 8,192, N = 4P: per point the device time of the step (CUDA
    events of the call, inputs in HBM), rounds, and decisions (one DECIDE per active prompt per
    round: n_q - n0 + 1 for every drawn prompt)."""
    import torch

    import paper_2607_26253_gb300 as pkg
    torch.cuda.set_device(0)
    P, B = 65536, 8192
    cfg = pkg.model_cfg(None, max_prompts=P, max_active=B, max_seqs=1, max_prompt_len=1, max_gen_len=1, max_k=16)
    rows = []
    with pkg.Handle(cfg, stream=torch.cuda.current_stream()) as h:
        for k in synth.SWEEP_K:
            for n0 in synth.SWEEP_N0:
                for tau in synth.SWEEP_TAU:
                    w = synth.sweep_workload(k, n0, tau)
                    si = synth.step_inputs(w)
                    thr = torch.from_numpy(si.thresholds.view(np.int64)).cuda()
                    lens = torch.from_numpy(si.lengths).cuda()
                    kw = dict(thresholds=thr, lengths=lens, N=w.budget_N, k=k, n0=n0, tau=tau, target_B=B,
                              reward_seed=w.reward_seed)
                    h.collect_step(**kw)  # warm-up
                    o = h.collect_step(**kw)
                    n = o.n.astype(np.int64)
                    dec = int((n[n > 0] - n0 + 1).sum())
                    rows.append((k, n0, tau, o.device_ms, o.counters["rounds"], dec))
    ms = np.array([r[3] for r in rows])
    rounds = np.array([r[4] for r in rows])
    dec = np.array([r[5] for r in rows])
    print(json.dumps({"metric": "controller microseconds per round / decisions per second (sweep, P = 65,536)",
                      "points": len(rows), "us_per_round_median": float(np.median(1e3 * ms / rounds)),
                      "us_per_round_max": float(np.max(1e3 * ms / rounds)),
                      "decisions_per_s_median": float(np.median(dec / (ms * 1e-3))),
                      "k8_n0_2_tau045": next({"ms": r[3], "rounds": r[4], "decisions": r[5]} for r in rows
                                            if r[0] == 8 and r[1] == 2 and abs(r[2] - 0.45) < 1e-9)}))


# --------------------------------------------------------------------------------- reference arm
def run_reference(args):
    """The oracle as the reference arm, on this host's cores: per step, O1 over the whole step's
    schedule and O2's teacher-forced slice (CPU_SLICE_STEPS decode steps of one round-0 rollout)
    on all host threads; value = decode tokens per second of O2."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from oracle import controller as oc
    w = synth.WORKLOADS[args.workload]
    o1 = []
    for i in range(args.steps):
        wi = w.with_seed_offset(7 * (args.warmup + i + 1))
        si = synth.step_inputs(wi)
        t0 = time.perf_counter()
        oc.collect_workload(wi, si)
        o1.append(time.perf_counter() - t0)
    secs = time_slice(args.workload, None, args.warmup + args.steps)[args.warmup:]
    value = CPU_SLICE_STEPS * len(secs) / sum(secs)
    try:
        avail = len(os.sched_getaffinity(0))
    except Exception:
        avail = os.cpu_count()
    sample = (f"per step: O1 over the whole step's schedule (1 thread) + O2 float64 teacher-forced slice, the "
              f"first {CPU_SLICE_STEPS} decode steps of one round-0 rollout by full recompute over the "
              f"{w.prompt_len}-token prompt, BLAS on all {avail} host threads; value = {CPU_SLICE_STEPS} / O2 time")
    line = {
        "impl": "reference",
        "metric": "rollout tokens/sec (also effective groups/sec and decode HBM GB/s)",
        "value": value, "unit": "tokens/s", "n_gpus": int(os.environ.get("WORLD_SIZE", "1")),
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * (sum(secs) + sum(o1)) / len(secs),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": {"workload": w.name},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": avail, "kind": "oracle", "sample": sample,
                         "cpu_model": cpu_model(), "o1_whole_step_s_mean": float(np.mean(o1))},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))


if __name__ == "__main__":
    a = parse()
    if a.cpu_slice:
        cpu_slice_child(a)
    elif a.kernel_profile is not None:
        run_kernel_profile(a)
    elif a.controller:
        run_controller(a)
    elif a.impl == "reference":
        run_reference(a)
    else:
        run_mine(a)
