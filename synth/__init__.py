"""Seeded synthetic workloads, shared as *inputs* by the CPU oracle and the CUDA path.

This module holds none of the method's arithmetic (no posterior, predictor,
decision rule, scheduler, attention or sampling): it only produces the seeded
inputs of the workloads the paper's experiments are shaped like (Sec. 4.1 and
App. E: B=64 prompts per step, k=8, n0=2, tau=0.45, 1.5B/3B decoder policies,
generation cap 4096), with random-init weights and synthetic rewards because
neither the datasets nor the trained weights are available.

Inputs produced here:
  * model weights, N(0, 0.02) rounded to bf16 (norm weights 1.0);
  * prompt tokens, uniform over the vocabulary;
  * each prompt's latent success rate p, from a mixture of point masses at 0
    and 1 and a Beta(2,2) component, delivered as the integer threshold
    floor(p * 2^32) (2^32 meaning "always succeeds");
  * each rollout's generated length L(q, j).
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
import threading
from dataclasses import dataclass, field, replace

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "_build", "libsynth.so")
_lock = threading.Lock()
_lib = None

GOLDEN = 0x9E3779B97F4A7C15
MASK64 = (1 << 64) - 1


def build(force: bool = False) -> str:
    """Compile synth/gen.c into synth/_build/libsynth.so (gcc, OpenMP)."""
    src = os.path.join(_HERE, "gen.c")
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(src)):
        return _LIB_PATH
    os.makedirs(os.path.dirname(_LIB_PATH), exist_ok=True)
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", "-O2", "-fPIC", "-shared", "-fopenmp", "-fno-fast-math",
                           "-o", tmp, src, "-lm"])
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            lib.synth_fill_normal_bf16.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint64,
                                                   ctypes.c_double, ctypes.c_void_p]
            lib.synth_fill_normal_bf16.restype = None
            lib.synth_fill_const_bf16.argtypes = [ctypes.c_uint64, ctypes.c_float, ctypes.c_void_p]
            lib.synth_fill_const_bf16.restype = None
            lib.synth_splitmix64_at.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
            lib.synth_splitmix64_at.restype = ctypes.c_uint64
            _lib = lib
    return _lib


# --------------------------------------------------------------------------------------------
# Shapes and workloads
# --------------------------------------------------------------------------------------------
@dataclass(frozen=True)
class ModelShape:
    """Decoder-only policy shape (pre-norm, RMSNorm, RoPE, GQA, SwiGLU, untied lm_head)."""
    name: str
    layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    vocab: int
    rope_theta: float = 1.0e6
    rms_eps: float = 1.0e-6

    @property
    def qkv_out(self) -> int:
        return (self.n_heads + 2 * self.n_kv_heads) * self.head_dim

    def layer_weight_bytes(self) -> int:
        d, f = self.d_model, self.ffn
        return 2 * (self.qkv_out * d + d * self.n_heads * self.head_dim + 2 * f * d + d * f)

    def kv_bytes_per_token(self) -> int:
        """bf16 K+V bytes one token occupies across all layers."""
        return self.layers * 2 * self.n_kv_heads * self.head_dim * 2


TINY = ModelShape("tiny-2L-d128", layers=2, d_model=128, n_heads=4, n_kv_heads=2, head_dim=32,
                  ffn=512, vocab=512)
SHAPE_1P5B = ModelShape("1.5B-shaped", layers=28, d_model=1536, n_heads=12, n_kv_heads=2,
                        head_dim=128, ffn=8960, vocab=151936)
SHAPE_3B = ModelShape("3B-shaped", layers=36, d_model=2048, n_heads=16, n_kv_heads=2, head_dim=128,
                      ffn=11008, vocab=151936)


@dataclass(frozen=True)
class Lengths:
    """Rollout-length law: 'uniform' on [lo, hi] or 'lognormal' with median/sigma, capped.
    hard_scale > 0 (lognormal only) ties length to difficulty: prompt q's median becomes
    median * (1 + hard_scale * (1 - p_q)), p_q its latent success rate, so the rollouts of
    all-fail prompts are the longest (hard_scale = 1: twice the all-pass median)."""
    kind: str
    lo: int = 1
    hi: int = 1
    median: float = 1.0
    sigma: float = 0.5
    cap: int = 1
    hard_scale: float = 0.0

    @property
    def max_len(self) -> int:
        return self.hi if self.kind == "uniform" else self.cap


@dataclass(frozen=True)
class Workload:
    """One RLVR step's rollout-collection problem (Algorithm 1's `Require` line)."""
    name: str
    model: ModelShape | None
    n_prompts: int            # pool size P (stream order = index)
    prompt_len: int           # Lp
    target_B: int
    k: int
    n0: int
    tau: float
    budget_N: int
    mixture: tuple = (0.35, 0.25, 0.40)   # P(p=0), P(p=1), P(p~Beta(2,2))
    lengths: Lengths = field(default_factory=lambda: Lengths("uniform", lo=8, hi=32))
    commit_min: int | None = None         # default k
    prior: tuple = (1, 1)                 # integer Beta prior (alpha0, beta0)
    seed_prompts: int = 1
    seed_latent: int = 2
    seed_lengths: int = 3
    reward_seed: int = 4
    sample_seed: int = 5
    weight_seed: int = 0

    @property
    def commit_floor(self) -> int:
        return self.k if self.commit_min is None else self.commit_min

    def with_seed_offset(self, off: int) -> "Workload":
        """Replicate: every seed shifted by `off` (weights stay the same policy)."""
        return replace(self, seed_prompts=self.seed_prompts + off, seed_latent=self.seed_latent + off,
                       seed_lengths=self.seed_lengths + off, reward_seed=self.reward_seed + off,
                       sample_seed=self.sample_seed + off)


WORKLOADS = {
    # 2-layer d=128 decoder; B=16 target from a 64-prompt stream (refill is exercised), N=128.
    "tiny": Workload("tiny: 2L d128, B=16, P=64x32 tok, k=8 n0=2 tau=.45 N=128", TINY,
                     n_prompts=64, prompt_len=32, target_B=16, k=8, n0=2, tau=0.45, budget_N=128,
                     lengths=Lengths("uniform", lo=8, hi=32)),
    "1.5b": Workload("1.5B-shaped: 28L d1536, B=64, P=256x256 tok, k=8 n0=2 tau=.45 N=512, "
                     "lognormal(1024, .5) cap 4096", SHAPE_1P5B,
                     n_prompts=256, prompt_len=256, target_B=64, k=8, n0=2, tau=0.45, budget_N=512,
                     lengths=Lengths("lognormal", median=1024, sigma=0.5, cap=4096)),
    "3b": Workload("3B-shaped: 36L d2048, B=64, P=256x384 tok, k=8 n0=2 tau=.45 N=512, "
                   "lognormal(1536, .5) cap 8192", SHAPE_3B,
                   n_prompts=256, prompt_len=384, target_B=64, k=8, n0=2, tau=0.45, budget_N=512,
                   lengths=Lengths("lognormal", median=1536, sigma=0.5, cap=8192)),
    "oversampled": Workload("oversampled pool at 1.5B shape: P=192, B=64, k=8 n0=2 tau=.45 "
                            "N=6Bk=3072, mixture 45/30/25, lognormal(2048, .5) cap 8192",
                            SHAPE_1P5B, n_prompts=192, prompt_len=256, target_B=64, k=8, n0=2,
                            tau=0.45, budget_N=3072, mixture=(0.45, 0.30, 0.25),
                            lengths=Lengths("lognormal", median=2048, sigma=0.5, cap=8192)),
}

SWEEP_K = (4, 8, 16)
SWEEP_N0 = (1, 2, 3)
SWEEP_TAU = (0.30, 0.35, 0.40, 0.45, 0.50, 0.55, 0.60)


def sweep_workload(k: int, n0: int, tau: float, replicate: int = 0, n_prompts: int = 65536,
                   target_B: int = 8192) -> Workload:
    """Controller-only sweep point: P=65,536 prompts, B=8192, N=4P, no decode."""
    w = Workload(f"controller sweep P={n_prompts} B={target_B} k={k} n0={n0} tau={tau:.2f} N=4P",
                 None, n_prompts=n_prompts, prompt_len=1, target_B=target_B, k=k, n0=n0, tau=tau,
                 budget_N=4 * n_prompts, lengths=Lengths("uniform", lo=1, hi=1))
    return w.with_seed_offset(100 * replicate)


# --------------------------------------------------------------------------------------------
# Generators
# --------------------------------------------------------------------------------------------
def splitmix64_at(seed: int, c: int) -> int:
    """Output number c (1-based) of SplitMix64 seeded with `seed` (Steele et al. 2014)."""
    z = (seed + c * GOLDEN) & MASK64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & MASK64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & MASK64
    return z ^ (z >> 31)


def latent_thresholds(w: Workload) -> np.ndarray:
    """uint64[P]: floor(p_q * 2^32) for each prompt's latent success rate p_q.

    p_q = 0 with prob mixture[0], 1 with prob mixture[1], else Beta(2,2) drawn
    as the median of three U(0,1) (the 2nd order statistic of 3 uniforms)."""
    rng = np.random.default_rng(w.seed_latent)
    P = w.n_prompts
    comp = rng.random(P)
    u3 = rng.random((P, 3))
    beta22 = np.median(u3, axis=1)
    p0, p1, _ = w.mixture
    p = np.where(comp < p0, 0.0, np.where(comp < p0 + p1, 1.0, beta22))
    thr = np.floor(p * 4294967296.0).astype(np.uint64)
    thr[p >= 1.0] = np.uint64(1 << 32)
    return thr


def constant_thresholds(P: int, gamma: float) -> np.ndarray:
    """uint64[P] with every prompt at success rate gamma (floor(gamma*2^32))."""
    t = np.uint64(1 << 32) if gamma >= 1.0 else np.uint64(int(math.floor(gamma * 4294967296.0)))
    return np.full(P, t, dtype=np.uint64)


def rollout_lengths(w: Workload) -> np.ndarray:
    """int32[P, k]: generated tokens of rollout j of prompt q."""
    rng = np.random.default_rng(w.seed_lengths)
    L = w.lengths
    shape = (w.n_prompts, w.k)
    if L.kind == "uniform":
        return rng.integers(L.lo, L.hi + 1, size=shape, dtype=np.int64).astype(np.int32)
    z = rng.standard_normal(shape)
    log_med = math.log(L.median)
    if L.hard_scale > 0:
        p = latent_thresholds(w).astype(np.float64) / 4294967296.0
        log_med = np.log(L.median * (1.0 + L.hard_scale * (1.0 - p)))[:, None]
    x = np.rint(np.exp(log_med + L.sigma * z))
    return np.clip(x, 1, L.cap).astype(np.int32)


def prompt_tokens(w: Workload) -> np.ndarray:
    """int32[P, Lp] uniform over the vocabulary."""
    rng = np.random.default_rng(w.seed_prompts)
    V = w.model.vocab if w.model is not None else 2
    return rng.integers(0, V, size=(w.n_prompts, w.prompt_len), dtype=np.int64).astype(np.int32)


# Per-tensor stream ids of the weight generator.
_T_ATTN_NORM, _T_WQ, _T_WK, _T_WV, _T_WO, _T_MLP_NORM, _T_WGATE, _T_WUP, _T_WDOWN = range(9)


def _normal_bf16(seed: int, stream: int, shape, std: float = 0.02) -> np.ndarray:
    out = np.empty(shape, dtype=np.uint16)
    _load().synth_fill_normal_bf16(seed, stream, out.size, std, out.ctypes.data)
    return out


def _ones_bf16(n: int) -> np.ndarray:
    out = np.empty(n, dtype=np.uint16)
    _load().synth_fill_const_bf16(n, 1.0, out.ctypes.data)
    return out


def layer_weights(m: ModelShape, layer: int, seed: int = 0) -> dict:
    """bf16 bit patterns (uint16) of one decoder layer, in [out_features, in_features] layout."""
    d, f, hd = m.d_model, m.ffn, m.head_dim
    base = 16 * (layer + 1)
    return {
        "attn_norm": _ones_bf16(d),
        "wq": _normal_bf16(seed, base + _T_WQ, (m.n_heads * hd, d)),
        "wk": _normal_bf16(seed, base + _T_WK, (m.n_kv_heads * hd, d)),
        "wv": _normal_bf16(seed, base + _T_WV, (m.n_kv_heads * hd, d)),
        "wo": _normal_bf16(seed, base + _T_WO, (d, m.n_heads * hd)),
        "mlp_norm": _ones_bf16(d),
        "wgate": _normal_bf16(seed, base + _T_WGATE, (f, d)),
        "wup": _normal_bf16(seed, base + _T_WUP, (f, d)),
        "wdown": _normal_bf16(seed, base + _T_WDOWN, (d, f)),
    }


def global_weights(m: ModelShape, seed: int = 0) -> dict:
    """Embedding [V, d], final norm [d], untied lm_head [V, d] (bf16 bits)."""
    return {
        "embed": _normal_bf16(seed, 1, (m.vocab, m.d_model)),
        "final_norm": _ones_bf16(m.d_model),
        "lm_head": _normal_bf16(seed, 2, (m.vocab, m.d_model)),
    }


def model_weights(m: ModelShape, seed: int = 0) -> dict:
    """All weights: {'embed','final_norm','lm_head','layers': [layer dicts]}."""
    g = global_weights(m, seed)
    g["layers"] = [layer_weights(m, l, seed) for l in range(m.layers)]
    return g


def bf16_bits_to_f32(a: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32."""
    return (a.astype(np.uint32) << 16).view(np.float32)


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even float32 -> bf16 bit patterns (finite inputs)."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)


@dataclass
class StepInputs:
    """Everything one rollout-collection step consumes besides the model."""
    workload: Workload
    thresholds: np.ndarray   # uint64[P]
    lengths: np.ndarray      # int32[P, k]
    tokens: np.ndarray | None  # int32[P, Lp] (None without a model)


def step_inputs(w: Workload) -> StepInputs:
    return StepInputs(w, latent_thresholds(w), rollout_lengths(w),
                      prompt_tokens(w) if w.model is not None else None)
