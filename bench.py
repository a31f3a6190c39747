"""Benchmark of one rollout-collection step (Algorithm 1 with batched bf16 decode) on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload 1.5b|3b|oversampled|tiny]
    python bench.py --impl reference ...      # the CPU oracle as the reference arm

A step is one sara_collect_step over a fresh synthetic prompt stream of the named workload:
probe, decide, refill and decode every issued rollout until the target or the budget is
reached.  `value` = rollout tokens generated per second over the K timed steps (inputs
resident in HBM), whole job over all ranks; `e2e` = the same metric through the same call
with host (pinned) inputs and host outputs, copies inside the timed region.  N > 1 runs one
replica per GPU on its own shard of the prompt stream (seed offset by rank, no collective
on the data path); only the final counters are reduced.

Rank 0 prints one JSON line.  Data are synthetic (random-init weights, seeded rewards).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

HERE_PEAKS = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_HBM_GBS = 6800.0


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="mine", choices=["mine", "reference"])
    ap.add_argument("--workload", default="1.5b", choices=sorted(synth.WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--kernel-profile", type=int, default=None, metavar="KERNEL",
                    help="profiling mode for ncu: launch one decode kernel (sara_profile ids; 0 = whole "
                         "eager decode step) on a reduced-capacity handle of the workload's shapes")
    ap.add_argument("--rows", type=int, default=25, help="live rows in --kernel-profile mode")
    ap.add_argument("--iters", type=int, default=5, help="launches in --kernel-profile mode")
    ap.add_argument("--ctx", type=int, default=None, help="context length in --kernel-profile mode "
                    "(default: prompt length + 128)")
    return ap.parse_args()


# --------------------------------------------------------------------------------- helpers
def peaks():
    try:
        with open(HERE_PEAKS) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


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


def decode_algorithmic_bytes(m: synth.ModelShape, Lp: int, lens: np.ndarray) -> float:
    """Bytes the decode of rollouts with generated lengths `lens` must move: every layer's
    weights + final norm + lm_head once per decode step is counted by the caller; here the
    per-token part: K/V reads of the whole context, K/V appends and embedding rows."""
    kvtok = m.kv_bytes_per_token()
    L = lens.astype(np.float64)
    ctx_sum = (L * Lp + L * (L - 1) / 2).sum()  # contexts Lp, Lp+1, .. Lp+L-1
    return ctx_sum * kvtok + L.sum() * kvtok + L.sum() * m.d_model * 2


def step_algorithmic_bytes(m: synth.ModelShape, rows: int, ctx: int) -> float:
    """Bytes one decode step over `rows` rows at context `ctx` must move: the weights once,
    the K/V of every context position read, the new K/V written, the embedding rows."""
    kvtok = m.kv_bytes_per_token()
    return weight_bytes_per_step(m) + rows * (ctx - 1) * kvtok + rows * kvtok + rows * m.d_model * 2


def weight_bytes_per_step(m: synth.ModelShape) -> int:
    return m.layers * (m.layer_weight_bytes() + 4 * m.d_model) + 2 * m.vocab * m.d_model + 2 * m.d_model


def executed_lengths(si, n: np.ndarray) -> np.ndarray:
    return np.concatenate([si.lengths[q, :int(n[q])] for q in range(len(n)) if n[q] > 0] or [np.zeros(0)])


# --------------------------------------------------------------------------------- CPU arm
def cpu_oracle_sample(w: synth.Workload, weights=None, tokens_per_sample: int = 1):
    """The oracle as it stands on this host's cores: the Algorithm 1 schedule of the whole
    step (O1) plus `tokens_per_sample` generated tokens of one rollout by full recompute (O2).
    Returns (tokens/s, seconds, description)."""
    from oracle import controller as oc
    from oracle import decode as o2
    si = synth.step_inputs(w)
    t0 = time.perf_counter()
    ref = oc.collect_workload(w, si)
    t1 = time.perf_counter()
    W = o2.Weights(w.model, weights)
    q = int(np.nonzero(ref.n)[0][0])
    t2 = time.perf_counter()
    o2.generate(W, si.tokens[q], tokens_per_sample, w.sample_seed, o2.uid_of(q, 0))
    t3 = time.perf_counter()
    per_token = (t3 - t2) / tokens_per_sample
    # whole-step cost model of the oracle: schedule + every generated token at this rate
    rate = 1.0 / per_token
    desc = (f"O1 schedule of the whole step ({t1 - t0:.3f} s) + O2 float64 decode of the first "
            f"{tokens_per_sample} token(s) of rollout (q={q}, j=0) by full recompute over the "
            f"{w.prompt_len}-token prompt; tokens/s = tokens / O2 time")
    return rate, (t1 - t0) + (t3 - t2), desc


# --------------------------------------------------------------------------------- GPU arm
def run_mine(args):
    import torch
    import torch.distributed as dist

    import paper_2607_26253_gb300 as pkg
    from paper_2607_26253_gb300 import replicas

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
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

    # one synthetic batch per step: a fresh prompt stream (seeds shifted by the step index)
    def inputs(i):
        wi = w.with_seed_offset(7 * (i + 1)) if i >= 0 else w
        return wi, synth.step_inputs(wi)

    def run_device(wi, si, dev_in):
        return h.collect_step(thresholds=dev_in[0], lengths=dev_in[1], tokens=dev_in[2], N=wi.budget_N, k=wi.k,
                              n0=wi.n0, tau=wi.tau, target_B=wi.target_B, reward_seed=wi.reward_seed,
                              sample_seed=wi.sample_seed, commit_min=wi.commit_floor, prior=wi.prior,
                              want_tokens=True, outputs_on_device=True)

    def to_dev(si):
        return (torch.from_numpy(si.thresholds.view(np.int64)).to(dev), torch.from_numpy(si.lengths).to(dev),
                torch.from_numpy(si.tokens).to(dev))

    batches = [inputs(i) for i in range(args.warmup + args.steps)]
    dev_batches = [to_dev(si) for _, si in batches]
    torch.cuda.synchronize(dev)
    for i in range(args.warmup):
        run_device(batches[i][0], batches[i][1], dev_batches[i])
    torch.cuda.synchronize(dev)

    # ------------------------------------------------------------------ timed region (HBM-resident)
    outs = []
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    with ClockSampler(local) as clk:
        e0.record(stream)
        for i in range(args.warmup, args.warmup + args.steps):
            outs.append(run_device(batches[i][0], batches[i][1], dev_batches[i]))
        e1.record(stream)
        torch.cuda.synchronize(dev)
    if world > 1:
        dist.barrier()
    ms = e0.elapsed_time(e1)
    clocks = clk.summary()

    tok = sum(o.counters["gen_tokens"] for o in outs)
    groups = sum(o.counters["committed"] for o in outs)
    rollouts = sum(o.counters["rollouts"] for o in outs)
    dsteps = sum(o.counters["decode_steps"] for o in outs)
    dec_bytes = 0.0
    for (wi, si), o in zip(batches[args.warmup:], outs):
        lens = executed_lengths(si, o.n.cpu().numpy())
        dec_bytes += decode_algorithmic_bytes(m, wi.prompt_len, lens) + o.counters["decode_steps"] * \
            weight_bytes_per_step(m)

    # ------------------------------------------------------------------ end to end (host buffers)
    def pinned(a):
        t = torch.empty(a.shape, dtype=torch.from_numpy(a[:0]).dtype, pin_memory=True)
        t.numpy()[...] = a
        return t.numpy()

    e2e_batches = []
    for i in range(args.steps):
        wi, si = inputs(args.warmup + args.steps + i)
        e2e_batches.append((wi, pinned(si.thresholds), pinned(si.lengths), pinned(si.tokens)))
    h2d = sum(b[1].nbytes + b[2].nbytes + b[3].nbytes for b in e2e_batches)
    d2h = 0
    e2e_tok = 0
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    f0.record(stream)
    for wi, thr, lens, toks in e2e_batches:
        o = h.collect_step(thresholds=thr, lengths=lens, tokens=toks, N=wi.budget_N, k=wi.k, n0=wi.n0, tau=wi.tau,
                           target_B=wi.target_B, reward_seed=wi.reward_seed, sample_seed=wi.sample_seed,
                           commit_min=wi.commit_floor, prior=wi.prior, want_tokens=True)
        e2e_tok += o.counters["gen_tokens"]
        d2h += o.status.nbytes + o.n.nbytes + o.s.nbytes + o.decided_round.nbytes + o.tokens.nbytes
    f1.record(stream)
    torch.cuda.synchronize(dev)
    e2e_ms = f0.elapsed_time(f1)

    # ------------------------------------------------------------------ dominant kernel roofline
    # the decode-step kernel (one launch = one whole forward over the live rows) at the
    # step's mean live rows and the median mid-rollout context
    mean_rows = max(1, int(round(tok / max(dsteps, 1))))
    mid_ctx = w.prompt_len + int(np.median(batches[0][1].lengths)) // 2
    k_ms = h.profile(1, mean_rows, mid_ctx, iters=20)
    k_bytes = step_algorithmic_bytes(m, mean_rows, mid_ctx)
    step_ms = h.profile(0, mean_rows, mid_ctx, iters=20)  # kernel + sampling / bookkeeping
    h.close()

    # ------------------------------------------------------------------ reduce over ranks
    if world > 1:  # the only collective: job totals (sum) over the slowest rank's time (max)
        ms, e2e_ms = replicas.reduce_max([ms, e2e_ms], device=dev)
        tok, groups, rollouts, e2e_tok, dec_bytes, h2d, d2h = replicas.reduce_sum(
            [tok, groups, rollouts, e2e_tok, dec_bytes, h2d, d2h], device=dev)
    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    peak, peak_kind = peaks()
    achieved = k_bytes / (k_ms * 1e-3) / 1e9
    # DRAM traffic of the capture, scaled to this launch by its algorithmic bytes (weights are
    # the same; KV grows with rows x context, which the capture read exactly once as well)
    tr = read_traffic(args.workload)
    traffic = None if tr is None else tr[0] * k_bytes / tr[1]
    cpu = None
    if not args.no_cpu_baseline:
        rate, secs, desc = cpu_oracle_sample(w0, weights)
        cpu = {"value": rate, "unit": "rollout tokens/s", "cores": os.cpu_count(), "kind": "oracle",
               "sample": desc, "seconds": round(secs, 2)}
    line = {
        "metric": "rollout tokens/sec (also effective groups/sec and decode HBM GB/s)",
        "value": tok / (ms * 1e-3),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms / args.steps,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (random-init weights N(0,0.02), seeded prompts, rewards and lengths)",
        "config": {"workload": w0.name, "global_batch": w0.target_B * world, "seq_len": w0.prompt_len,
                   "parallelism": f"replicas x{world} (prompt-stream shards)",
                   "l2": "inputs larger than L2 (3+ GB of weights streamed per decode step)"},
        "effective_groups_per_s": groups / (ms * 1e-3),
        "rollouts_per_s": rollouts / (ms * 1e-3),
        "decode_hbm_gbs": dec_bytes / (ms * 1e-3) / 1e9,
        "decode_hbm_frac": dec_bytes / (ms * 1e-3) / 1e9 / peak,
        "decode_step_ms": step_ms,
        "decode_kernel_ms": k_ms,
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic,
                     "traffic_note": None if tr is None else "ncu capture at 25 rows, context 384, scaled by algorithmic bytes",
                     "kernel": f"decode_step_kernel (whole forward), {mean_rows} live rows at context {mid_ctx}",
                     "bytes_per_launch": k_bytes,
                     "peak_kind": f"{peak_kind} burst copy"},
        "e2e": {"value": e2e_tok / (e2e_ms * 1e-3), "unit": "tokens/s", "h2d_bytes_per_step": h2d / args.steps,
                "d2h_bytes_per_step": d2h / args.steps},
        "cpu_baseline": cpu,
        "gpu_launches": None,
        "clocks": clocks,
    }
    # kernels launched: per decode step the controller, the decode-step kernel and the
    # sampling/bookkeeping kernel; per round start the prefill (embedding + 5 per layer
    # but the last layer's 4) and the KV fan-out; per call the init kernel
    rounds = sum(o.counters["rounds"] for o in outs)
    line["gpu_launches"] = int(3 * dsteps + rounds * (1 + 5 * m.layers - 4 + 1) + args.steps)
    print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()


def read_traffic(workload: str):
    """(DRAM bytes, algorithmic bytes) of one launch of the dominant kernel from the committed
    ncu summary, or None."""
    path = os.path.join(ROOT, "profiles", f"decode_step_{workload.replace('.', 'p')}_ncu.md")
    got = {}
    try:
        for line in open(path):
            for key in ("traffic_bytes_per_launch:", "algorithmic_bytes_per_launch:"):
                if line.startswith(key):
                    got[key] = float(line.split(":", 1)[1].split()[0])
    except OSError:
        return None
    if len(got) != 2:
        return None
    return got["traffic_bytes_per_launch:"], got["algorithmic_bytes_per_launch:"]


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
    with pkg.Handle(cfg, weights, stream=torch.cuda.current_stream()) as h:
        ms = h.profile(args.kernel_profile, args.rows, ctx, iters=args.iters)
    print(json.dumps({"kernel": args.kernel_profile, "rows": args.rows, "ctx": ctx, "ms_per_launch": ms}))


# --------------------------------------------------------------------------------- reference arm
def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    w = synth.WORKLOADS[args.workload]
    weights = synth.model_weights(w.model, w.weight_seed)
    for _ in range(args.warmup):
        cpu_oracle_sample(w, weights)
    rates, secs = [], 0.0
    desc = ""
    for _ in range(args.steps):
        r, s, desc = cpu_oracle_sample(w, weights)
        rates.append(r)
        secs += s
    value = float(np.mean(rates))
    line = {
        "impl": "reference",
        "metric": "rollout tokens/sec (also effective groups/sec and decode HBM GB/s)",
        "value": value, "unit": "tokens/s", "n_gpus": int(os.environ.get("WORLD_SIZE", "1")),
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * secs / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": {"workload": w.name},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
                         "sample": desc},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))


if __name__ == "__main__":
    a = parse()
    if a.kernel_profile is not None:
        run_kernel_profile(a)
    elif a.impl == "reference":
        run_reference(a)
    else:
        run_mine(a)
