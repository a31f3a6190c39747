"""O1w -- the SARA step with the history warm-start (spec oracle).

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).  The paper's optional warm-start carries each
prompt's Beta posterior from one RLVR step to the next with an exponential decay lambda, so a
prompt seen saturated at the last step starts skewed and is abandoned after fewer probes (App. D,
"Defaults and history warm-start"; the prior of Sec. 3.2 then comes from history).  The priors
become real numbers, so the effectiveness predictor of Prop. 1 / Eq. (peff) is evaluated in
float64 through log-Gamma and Eq. (decide) compares it with tau_low in float64.

Readings (the paper states the idea, not a formula):
- the carried state of a prompt is its decayed evidence on top of the base prior (alpha0, beta0):
  after a step that used prior (a, b) and observed n rollouts with s successes,
      a' = alpha0 + lambda * (a - alpha0 + s),    b' = beta0 + lambda * (b - beta0 + n - s)
  (an undrawn prompt has n = s = 0 and decays toward the base prior); lambda = 0 is plain SARA,
  lambda = 1 accumulates every observation;
- within a step everything is Algorithm 1 as in O1 (round-synchronous, continuing prompts funded
  first by p_eff, then whole n0-probes toward B - |C|), with each prompt's own prior; priority ties
  are broken by stream index.
"""
from __future__ import annotations

import math

import numpy as np

from . import controller as oc


def log_beta(x: float, y: float) -> float:
    return math.lgamma(x) + math.lgamma(y) - math.lgamma(x + y)


def peff(n: int, s: int, k: int, a: float, b: float) -> float:
    """Eq. (peff) with a real prior Beta(a, b): probability that the completed group of k is mixed
    given n rollouts with s successes (posterior Beta(a + s, b + n - s))."""
    if 0 < s < n:
        return 1.0
    ap, bp, r = a + s, b + (n - s), k - n
    out = 1.0
    if s == 0:   # every remaining rollout fails
        out -= math.exp(log_beta(ap, bp + r) - log_beta(ap, bp))
    if s == n:   # every remaining rollout succeeds
        out -= math.exp(log_beta(ap + r, bp) - log_beta(ap, bp))
    return out


def decide(n: int, s: int, k: int, tau: float, commit_min: int, a: float, b: float) -> int:
    """Eq. (decide) in the rule order of O1: commit a mixed group of at least commit_min, abandon
    at n = k (all-same there) or when p_eff < tau_low, else continue."""
    if 0 < s < n and n >= commit_min:
        return oc.COMMIT
    if n == k:
        return oc.ABANDON
    if peff(n, s, k, a, b) < tau:
        return oc.ABANDON
    return oc.CONTINUE


def carry(prior_a: np.ndarray, prior_b: np.ndarray, n: np.ndarray, s: np.ndarray, alpha0: float, beta0: float,
          lam: float):
    """The next step's priors from this step's priors and observations (the reading above)."""
    n = n.astype(np.float64)
    s = s.astype(np.float64)
    return (alpha0 + lam * (prior_a - alpha0 + s), beta0 + lam * (prior_b - beta0 + (n - s)))


def collect_step(thresholds: np.ndarray, lengths: np.ndarray, prior_a: np.ndarray, prior_b: np.ndarray, *,
                 k: int, n0: int, tau: float, target_B: int, N: int, reward_seed: int = 0,
                 commit_min: int | None = None, prompt_len: int = 1) -> oc.StepResult:
    """Algorithm 1 with a per-prompt real prior (a_q, b_q); outputs as O1's collect_step."""
    thr = np.ascontiguousarray(thresholds, dtype=np.uint64)
    P = thr.size
    cm = k if commit_min is None else commit_min
    L = np.asarray(lengths, dtype=np.int64)
    v = oc.verdicts(thr, k, reward_seed)
    a = np.asarray(prior_a, dtype=np.float64)
    b = np.asarray(prior_b, dtype=np.float64)
    status = np.full(P, oc.UNDRAWN, np.uint8)
    n = np.zeros(P, np.int64)
    s = np.zeros(P, np.int64)
    rnd = np.full(P, -1, np.int16)
    used = gen = steps = rounds = drawn = 0
    C = cursor = 0
    active, issued = [], []

    def draw():
        nonlocal cursor, used, drawn
        while cursor < P and len(active) < target_B - C and used + n0 <= N:
            q = cursor
            cursor += 1
            status[q] = oc.ACTIVE
            active.append(q)
            issued.append((q, n0))
            used += n0
            drawn += 1

    draw()
    rnd_i = 0
    ipr = []
    while issued:
        maxL = 0
        count = 0
        for q, c in issued:          # execute the round
            for _ in range(c):
                j = int(n[q])
                s[q] += int(v[q, j])
                n[q] += 1
                gen += int(L[q, j])
                maxL = max(maxL, int(L[q, j]))
                count += 1
        ipr.append(count)
        steps += maxL
        rounds += 1
        keep = []
        for q in active:             # DECIDE in stream order
            d = decide(int(n[q]), int(s[q]), k, tau, cm, float(a[q]), float(b[q]))
            if d == oc.COMMIT:
                status[q] = oc.COMMITTED
                rnd[q] = rnd_i
                C += 1
            elif d == oc.ABANDON:
                status[q] = oc.ABANDONED
                rnd[q] = rnd_i
            else:
                keep.append(q)
        active = keep
        issued = []
        if C >= target_B:
            break
        prio = sorted(active, key=lambda q: (-peff(int(n[q]), int(s[q]), k, float(a[q]), float(b[q])), q))
        for q in prio:               # continuing prompts first, by p_eff
            if used + 1 <= N:
                issued.append((q, 1))
                used += 1
            else:
                status[q] = oc.INCOMPLETE
        active = [q for q in active if status[q] == oc.ACTIVE]
        draw()                       # then fresh probes toward B - |C|
        rnd_i += 1
    for q in active:
        if status[q] == oc.ACTIVE:
            status[q] = oc.INCOMPLETE
    counters = {"rollouts": used, "gen_tokens": gen, "prefill_tokens": drawn * (prompt_len - 1),
                "decode_steps": steps, "rounds": rounds, "committed": int((status == oc.COMMITTED).sum()),
                "abandoned": int((status == oc.ABANDONED).sum()), "incomplete": int((status == oc.INCOMPLETE).sum()),
                "prompts_drawn": drawn}
    return oc.StepResult(status, n.astype(np.uint8), s.astype(np.uint8), rnd, counters, np.array(ipr, np.int32))
