"""O1 -- Python face of the C controller oracle (oracle/controller.c).

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).  Algorithm 1 of arxiv
2607.26253 (round-synchronous SARA step) with the closed-form predictor of
Prop. 1 / Eq. (peff) and the threshold rule of Eq. (decide), decided in exact
rational arithmetic.
"""
from __future__ import annotations

import ctypes
from dataclasses import dataclass
from fractions import Fraction

import numpy as np

from . import build

UNDRAWN, ACTIVE, COMMITTED, ABANDONED, INCOMPLETE = range(5)
CONTINUE, COMMIT, ABANDON = range(3)
COUNTER_NAMES = ("rollouts", "gen_tokens", "prefill_tokens", "decode_steps", "rounds",
                 "committed", "abandoned", "incomplete", "prompts_drawn")

_lib = None


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        lib.o1_collect_step.argtypes = [
            ctypes.c_int32, P, P, P, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int64,
            ctypes.c_int64,
            ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int64,
            ctypes.c_uint64, P, P, P, P, P, P, ctypes.c_int32]
        lib.o1_collect_step.restype = ctypes.c_int
        lib.o1_peff.argtypes = [ctypes.c_int] * 5 + [P]
        lib.o1_peff.restype = ctypes.c_int
        lib.o1_decide.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int64,
                                  ctypes.c_int64, ctypes.c_int, ctypes.c_int, ctypes.c_int]
        lib.o1_decide.restype = ctypes.c_int
        lib.o1_verdicts.argtypes = [ctypes.c_int64, ctypes.c_int32, P, ctypes.c_uint64, P]
        lib.o1_verdicts.restype = None
        _lib = lib
    return _lib


@dataclass
class StepResult:
    status: np.ndarray         # uint8[P]
    n: np.ndarray              # uint8[P] rollouts spent on each prompt
    s: np.ndarray              # uint8[P] successes observed
    decided_round: np.ndarray  # int16[P], -1 unless committed / abandoned
    counters: dict
    issued_per_round: np.ndarray


def peff(n: int, s: int, k: int, alpha0: int = 1, beta0: int = 1) -> Fraction:
    """Exact p_eff(n, s) from the C oracle."""
    out = np.zeros(4, dtype=np.uint64)
    rc = _load().o1_peff(n, s, k, alpha0, beta0, out.ctypes.data)
    if rc != 0:
        raise ValueError("invalid p_eff arguments")
    num = (int(out[0]) << 64) | int(out[1])
    den = (int(out[2]) << 64) | int(out[3])
    return Fraction(num, den)


def tau_fraction(tau) -> Fraction:
    """tau_low as an exact rational: a Fraction as given, a float by its shortest decimal
    (0.45 -> 9/20), matching how the paper states its thresholds."""
    f = tau if isinstance(tau, Fraction) else Fraction(repr(float(tau)))
    if not (0 <= f <= 1) or f.denominator > 2147483647:
        raise ValueError(f"tau_low must be a rational in [0, 1] with a 31-bit denominator: {tau}")
    return f


def decide(n: int, s: int, k: int, tau, commit_min: int | None = None, alpha0: int = 1,
           beta0: int = 1) -> int:
    """DECIDE(n, s) of Eq. (decide): CONTINUE, COMMIT or ABANDON."""
    t = tau_fraction(tau)
    r = _load().o1_decide(n, s, k, t.numerator, t.denominator,
                          k if commit_min is None else commit_min, alpha0, beta0)
    if r < 0:
        raise ValueError("invalid DECIDE arguments")
    return r


def verdicts(thresholds: np.ndarray, k: int, reward_seed: int) -> np.ndarray:
    """uint8[P, k]: the synthetic Bernoulli verdict of every (prompt, rollout index)."""
    thr = np.ascontiguousarray(thresholds, dtype=np.uint64)
    out = np.empty((thr.size, k), dtype=np.uint8)
    _load().o1_verdicts(thr.size, k, thr.ctypes.data, reward_seed, out.ctypes.data)
    return out


def collect_step(thresholds: np.ndarray | None, lengths: np.ndarray | None, *, k: int, n0: int,
                 tau, target_B: int, N: int, reward_seed: int = 0,
                 commit_min: int | None = None, prior=(1, 1), prompt_len: int = 1,
                 verdict_table: np.ndarray | None = None, n_prompts: int | None = None,
                 max_rounds: int = 4096) -> StepResult:
    """Run Algorithm 1 over a prompt stream and return every prompt's outcome."""
    if thresholds is not None:
        thr = np.ascontiguousarray(thresholds, dtype=np.uint64)
        P = thr.size
    else:
        thr = None
        P = int(n_prompts if n_prompts is not None else verdict_table.shape[0])
    lens = None if lengths is None else np.ascontiguousarray(lengths, dtype=np.int32)
    vt = None if verdict_table is None else np.ascontiguousarray(verdict_table, dtype=np.uint8)
    status = np.zeros(P, np.uint8)
    n = np.zeros(P, np.uint8)
    s = np.zeros(P, np.uint8)
    rnd = np.zeros(P, np.int16)
    counters = np.zeros(len(COUNTER_NAMES), np.int64)
    ipr = np.zeros(max_rounds, np.int32)
    ptr = lambda a: None if a is None else a.ctypes.data
    t = tau_fraction(tau)
    rc = _load().o1_collect_step(
        P, ptr(thr), ptr(lens), ptr(vt), prompt_len, k, n0, t.numerator, t.denominator,
        k if commit_min is None else commit_min, prior[0], prior[1], target_B, N, reward_seed,
        status.ctypes.data, n.ctypes.data, s.ctypes.data, rnd.ctypes.data, counters.ctypes.data,
        ipr.ctypes.data, max_rounds)
    if rc != 0:
        raise ValueError(f"o1_collect_step rejected its arguments (rc={rc})")
    c = {name: int(v) for name, v in zip(COUNTER_NAMES, counters)}
    return StepResult(status, n, s, rnd, c, ipr[:c["rounds"]].copy())


def collect_workload(w, si=None) -> StepResult:
    """Algorithm 1 on a synth.Workload's seeded inputs."""
    import synth
    si = si if si is not None else synth.step_inputs(w)
    return collect_step(si.thresholds, si.lengths, k=w.k, n0=w.n0, tau=w.tau, target_B=w.target_B,
                        N=w.budget_N, reward_seed=w.reward_seed, commit_min=w.commit_floor,
                        prior=w.prior, prompt_len=w.prompt_len)
