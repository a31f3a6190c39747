"""O1a -- the asynchronous per-prompt variant of the SARA step (spec oracle).

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).  The paper runs Algorithm 1 in synchronised
rounds and names the round barrier as a limitation (Discussion, Limitations (ii)).  This is the
variant without the barrier, in step-granular decode time; everything else is Algorithm 1 with
the closed-form predictor of Prop. 1 / Eq. (peff) and the rule of Eq. (decide):

- A rollout of length L that starts at decode step t0 occupies steps t0 .. t0 + L - 1.
  A prompt has at most one batch in flight (its n0-rollout probe, or the one rollout of a
  continue decision); it is decided at the end of the step in which that batch's last rollout
  finishes, instead of at the end of a round.
- At the end of a step, the prompts decided there follow the round rules of the synchronous
  oracle, as if they were one round:
  - DECIDE in stream order;
  - stop issuing once |C| >= B;
  - otherwise fund the continuing ones with one rollout each, highest p_eff first (ties: lower
    stream index), while the budget allows, the rest ending INCOMPLETE;
  - then draw fresh prompts in stream order while fewer than B - |C| prompts are in flight and
    a whole n0-probe fits the budget.
  New rollouts start at the next step.
- No cancellation: after the stop, rollouts in flight run to completion and their prompts are
  decided (commits past B are kept, a continue becomes INCOMPLETE).
- reserve=True (an alternative reading): a fresh prompt is drawn only if the budget covers it
  and every prompt in flight running to k rollouts, so a continue decision is always funded and
  continuing prompts keep first call on the budget as in the round rules.  The equal-length
  equivalence below holds for reserve=False only.

With every rollout length equal, all prompts in flight finish in the same step, so this
schedule reproduces the round-synchronous oracle exactly (decode steps = rounds x L).

prior_a / prior_b (optional, float64 [P]): the history warm-start (App. D) on this schedule --
each prompt's own real Beta prior in Eq. (peff) and Eq. (decide) and in the priority of
continuing prompts, evaluated in float64 exactly as the warm-start oracle O1w does
(oracle/warm_start.py); with equal lengths the schedule then reproduces O1w's round-synchronous
step.
"""
from __future__ import annotations

import heapq
from dataclasses import dataclass

import numpy as np

from . import controller as oc
from . import warm_start as ow

COUNTER_NAMES = ("rollouts", "gen_tokens", "prefill_tokens", "decode_steps", "events",
                 "committed", "abandoned", "incomplete", "prompts_drawn")


@dataclass
class AsyncResult:
    status: np.ndarray        # uint8[P], the controller's status codes
    n: np.ndarray             # uint8[P] rollouts spent on each prompt
    s: np.ndarray             # uint8[P] successes observed
    decided_step: np.ndarray  # int32[P]: end of the decode step of the commit / abandon, else -1
    decided_event: np.ndarray  # int32[P]: index of that step boundary among those with decisions
    counters: dict

    @property
    def mean_live_rollouts(self) -> float:
        """Rollouts in flight per decode step (every one of them decodes one token per step)."""
        d = self.counters["decode_steps"]
        return self.counters["gen_tokens"] / d if d else 0.0


def collect_step(thresholds: np.ndarray, lengths: np.ndarray, *, k: int, n0: int, tau, target_B: int,
                 N: int, reward_seed: int = 0, commit_min: int | None = None, prior=(1, 1),
                 prompt_len: int = 1, reserve: bool = False, prior_a=None, prior_b=None) -> AsyncResult:
    thr = np.ascontiguousarray(thresholds, dtype=np.uint64)
    P = thr.size
    L = np.ascontiguousarray(lengths, dtype=np.int64)
    if L.shape != (P, k) or (P and L.min() < 1):
        raise ValueError("lengths must be [P][k] with every length >= 1")
    if not (1 <= n0 <= k) or target_B < 1 or N < 0:
        raise ValueError("invalid step parameters")
    cm = k if commit_min is None else commit_min
    a0, b0 = prior
    v = oc.verdicts(thr, k, reward_seed)  # uint8[P][k]: rollout j of prompt q
    if (prior_a is None) != (prior_b is None):
        raise ValueError("prior_a and prior_b go together")
    if prior_a is not None:  # per-prompt real priors (warm-start): float64 predictor and rule
        pa = np.asarray(prior_a, dtype=np.float64)
        pb = np.asarray(prior_b, dtype=np.float64)

        def decide(q, nn, ss):
            return ow.decide(nn, ss, k, float(tau), cm, float(pa[q]), float(pb[q]))

        def peff(q):
            return ow.peff(int(n[q]), int(s[q]), k, float(pa[q]), float(pb[q]))
    else:
        def decide(q, nn, ss):
            return oc.decide(nn, ss, k, tau, cm, a0, b0)

        def peff(q):
            return oc.peff(int(n[q]), int(s[q]), k, a0, b0)

    status = np.full(P, oc.UNDRAWN, np.uint8)
    n = np.zeros(P, np.int64)
    s = np.zeros(P, np.int64)
    decided = np.full(P, -1, np.int32)
    decided_ev = np.full(P, -1, np.int32)
    batch = {}  # q -> rollouts of its batch in flight
    heap = []   # (decision step, q)
    used = tokens = drawn = 0
    C = 0
    cursor = 0
    stopped = False
    last_step = -1
    events = 0

    def issue(q: int, c: int, start: int) -> None:
        nonlocal used, tokens
        js = range(int(n[q]), int(n[q]) + c)
        batch[q] = c
        used += c
        tokens += int(sum(L[q, j] for j in js))
        heapq.heappush(heap, (start + int(max(L[q, j] for j in js)) - 1, q))

    def reserved() -> int:  # rollouts the prompts in flight may still take (reserve=True)
        return sum(k - int(n[q]) - c for q, c in batch.items()) if reserve else 0

    def draw(start: int) -> None:
        nonlocal cursor, drawn
        while cursor < P and len(batch) < target_B - C and used + (k if reserve else n0) + reserved() <= N:
            q = cursor
            cursor += 1
            status[q] = oc.ACTIVE
            drawn += 1
            issue(q, n0, start)

    draw(0)
    while heap:
        t = heap[0][0]
        done = []
        while heap and heap[0][0] == t:
            done.append(heapq.heappop(heap)[1])
        done.sort()
        ev = events
        events += 1
        last_step = t
        cont = []
        for q in done:  # the batch's verdicts, then DECIDE in stream order
            c = batch.pop(q)
            s[q] += int(v[q, n[q]:n[q] + c].sum())
            n[q] += c
            d = decide(q, int(n[q]), int(s[q]))
            if d == oc.COMMIT:
                status[q] = oc.COMMITTED
                decided[q] = t
                decided_ev[q] = ev
                C += 1
            elif d == oc.ABANDON:
                status[q] = oc.ABANDONED
                decided[q] = t
                decided_ev[q] = ev
            else:
                cont.append(q)
        if stopped or C >= target_B:
            stopped = True
            for q in cont:
                status[q] = oc.INCOMPLETE
            continue
        prio = sorted(cont, key=lambda q: (-peff(q), q))
        for q in prio:
            if used + 1 <= N:
                issue(q, 1, t + 1)
            else:
                status[q] = oc.INCOMPLETE
        draw(t + 1)

    counters = {
        "rollouts": used, "gen_tokens": tokens, "prefill_tokens": drawn * (prompt_len - 1),
        "decode_steps": last_step + 1, "events": events,
        "committed": int((status == oc.COMMITTED).sum()), "abandoned": int((status == oc.ABANDONED).sum()),
        "incomplete": int((status == oc.INCOMPLETE).sum()), "prompts_drawn": drawn,
    }
    return AsyncResult(status, n.astype(np.uint8), s.astype(np.uint8), decided, decided_ev, counters)


def collect_workload(w, si=None, reserve: bool = False) -> AsyncResult:
    """The asynchronous schedule on a synth.Workload's seeded inputs."""
    import synth
    si = si if si is not None else synth.step_inputs(w)
    return collect_step(si.thresholds, si.lengths, k=w.k, n0=w.n0, tau=w.tau, target_B=w.target_B,
                        N=w.budget_N, reward_seed=w.reward_seed, commit_min=w.commit_floor,
                        prior=w.prior, prompt_len=w.prompt_len, reserve=reserve)
