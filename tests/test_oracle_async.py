"""Pins of the asynchronous per-prompt schedule oracle (oracle/async_schedule.py).

- With every rollout length equal it must reproduce the round-synchronous oracle exactly (every
  prompt in flight finishes in the same step, so each step boundary is a round).
- With random lengths, invariants that hold by construction of Algorithm 1 plus the event rule,
  checked against quantities recomputed here from the verdict and length tables.
- The schedule's effect on the 1.5B-shaped workload (fewer decode steps, more rollouts in flight).
"""
from dataclasses import replace

import numpy as np
import pytest

import synth
from oracle import async_schedule as oa
from oracle import controller as oc


def _random_case(rng, it):
    k = int(rng.integers(2, 17))
    n0 = int(rng.integers(1, k + 1))
    P = int(rng.integers(1, 400))
    B = int(rng.integers(1, P + 1))
    w = synth.Workload("async", None, n_prompts=P, prompt_len=int(rng.integers(1, 5)), target_B=B, k=k, n0=n0,
                       tau=float(rng.choice([0.0, 0.3, 0.45, 0.6, 1.0])), budget_N=int(rng.integers(0, 4 * P * k // 2 + 1)),
                       commit_min=int(rng.integers(2, k + 1)), prior=(int(rng.integers(1, 9)), int(rng.integers(1, 9))),
                       lengths=synth.Lengths("uniform", lo=1, hi=60), seed_latent=it, seed_lengths=it + 1,
                       reward_seed=it + 2)
    return w, synth.step_inputs(w)


def test_equal_lengths_reproduce_the_round_synchronous_oracle():
    rng = np.random.default_rng(11)
    for it in range(120):
        w, si = _random_case(rng, it)
        Lc = int(rng.integers(1, 50))
        lengths = np.full_like(si.lengths, Lc)
        kw = dict(k=w.k, n0=w.n0, tau=w.tau, target_B=w.target_B, N=w.budget_N, reward_seed=w.reward_seed,
                  commit_min=w.commit_floor, prior=w.prior, prompt_len=w.prompt_len)
        sync = oc.collect_step(si.thresholds, lengths, **kw)
        asy = oa.collect_step(si.thresholds, lengths, **kw)
        assert np.array_equal(asy.status, sync.status), it
        assert np.array_equal(asy.n, sync.n) and np.array_equal(asy.s, sync.s), it
        dec = sync.decided_round >= 0
        assert np.array_equal(asy.decided_step >= 0, dec)
        assert np.array_equal(asy.decided_step[dec], (sync.decided_round[dec].astype(np.int64) + 1) * Lc - 1)
        assert np.array_equal(asy.decided_event, sync.decided_round.astype(np.int32))
        for key in ("rollouts", "gen_tokens", "prefill_tokens", "committed", "abandoned", "incomplete",
                    "prompts_drawn"):
            assert asy.counters[key] == sync.counters[key], (it, key)
        assert asy.counters["events"] == sync.counters["rounds"]
        assert asy.counters["decode_steps"] == sync.counters["rounds"] * Lc


@pytest.mark.parametrize("reserve", [False, True])
def test_invariants_with_random_lengths(reserve):
    rng = np.random.default_rng(12)
    for it in range(120):
        w, si = _random_case(rng, it)
        r = oa.collect_workload(w, si, reserve=reserve)
        k, N, B = w.k, w.budget_N, w.target_B
        v = oc.verdicts(si.thresholds, k, w.reward_seed).astype(np.int64)
        drawn = r.counters["prompts_drawn"]
        st = r.status
        n = r.n.astype(np.int64)
        # prompts are drawn in stream order, each with its whole probe
        assert np.all(st[:drawn] != oc.UNDRAWN) and np.all(st[drawn:] == oc.UNDRAWN)
        assert np.all(n[:drawn] >= w.n0) and np.all(n <= k)
        # successes and tokens are those of each prompt's first n rollouts
        assert all(int(r.s[q]) == int(v[q, :n[q]].sum()) for q in range(drawn))
        assert r.counters["gen_tokens"] == sum(int(si.lengths[q, :n[q]].sum()) for q in range(drawn))
        assert r.counters["rollouts"] == int(n.sum()) <= N
        # every decision is Eq. (decide) at the prompt's final counts
        for q in np.flatnonzero((st == oc.COMMITTED) | (st == oc.ABANDONED)):
            d = oc.decide(int(n[q]), int(r.s[q]), k, w.tau, w.commit_floor, *w.prior)
            assert d == (oc.COMMIT if st[q] == oc.COMMITTED else oc.ABANDON)
            assert 0 <= r.decided_step[q] < r.counters["decode_steps"]
        for q in np.flatnonzero(st == oc.INCOMPLETE):
            assert oc.decide(int(n[q]), int(r.s[q]), k, w.tau, w.commit_floor, *w.prior) == oc.CONTINUE
        # the step's last decode step is when its last batch finished
        assert (r.counters["decode_steps"] == 0) == (drawn == 0)
        if reserve and r.counters["committed"] < B:
            assert r.counters["incomplete"] == 0  # continuing prompts always funded


def test_async_schedule_on_the_1p5b_workload():
    # the schedule without the round barrier: fewer decode steps, more rollouts decoding at once
    w = synth.WORKLOADS["1.5b"]
    steps = np.zeros(3)
    live = np.zeros(3)
    comm = np.zeros(3)
    inc = np.zeros(3)
    for rep in range(4):
        wi = w.with_seed_offset(7 * (rep + 1))
        si = synth.step_inputs(wi)
        res = [oc.collect_workload(wi, si), oa.collect_workload(wi, si), oa.collect_workload(wi, si, reserve=True)]
        for i, r in enumerate(res):
            c = r.counters
            steps[i] += c["decode_steps"]
            live[i] += c["gen_tokens"] / c["decode_steps"]
            comm[i] += c["committed"]
            inc[i] += c["incomplete"]
    assert steps[1] < 0.6 * steps[0] and live[1] > 1.8 * live[0]
    # at this binding budget the plain asynchronous refill spends the budget on fresh probes
    # and leaves groups INCOMPLETE; with the reservation no group is left without funding
    assert inc[1] > inc[0] and inc[2] == 0 and comm[2] > comm[0]


def test_async_schedule_when_the_budget_does_not_bind():
    w = synth.WORKLOADS["oversampled"]
    si = synth.step_inputs(w)
    sync = oc.collect_workload(w, si)
    for reserve in (False, True):
        asy = oa.collect_workload(w, si, reserve=reserve)
        assert asy.counters["committed"] == sync.counters["committed"]
        assert asy.counters["decode_steps"] < 0.5 * sync.counters["decode_steps"]


# --------------------------------------------------------------------------------------------
# Hand-worked cases with unequal lengths.  Every verdict is fixed by the thresholds (0: every
# rollout fails), tau = 0 and commit floor 2, so a group is never abandoned before n = k (rule
# (iii) needs p_eff < 0) and, all-fail, it continues one rollout at a time with
# p_eff(n, 0) = (k - n) / (k + 1) (Prop. 1): 0.4 at n = 2, 0.2 at n = 3 for k = 4.  A batch
# started at step t0 with lengths L occupies steps t0 .. t0 + max L - 1; the prompt is decided at
# the end of that step; new rollouts start at the next step.
def _hand_case(lengths, P, B, N):
    thr = np.zeros(P, np.uint64)
    return oa.collect_step(thr, np.array(lengths, np.int32), k=4, n0=2, tau=0.0, target_B=B, N=N,
                           reward_seed=9, commit_min=2)


def test_hand_worked_ties_budget_and_next_step_start():
    # q0 [3,1,2,5], q1 [1,1,4,1], q2 [2,2,1,1]; B = 2, N = 9.
    # step 0: draw q0 (probe ends step 2, used 2), q1 (ends step 0, used 4); 2 in flight.
    # end of 0: q1 n=2 -> continue, funded (used 5): j=2 (L=4) runs steps 1..4.
    # end of 2: q0 n=2 -> continue, funded (used 6): j=2 (L=2) runs steps 3..4.
    # end of 4: q0 and q1 both n=3, p_eff 0.2 each: tie -> stream order; q0 j=3 (L=5) runs
    #           5..9 (used 7), q1 j=3 (L=1) runs 5..5 (used 8).
    # end of 5: q1 n=4 all-fail -> ABANDON (event 3); a fresh probe needs 10 > 9: q2 not drawn.
    # end of 9: q0 n=4 -> ABANDON (event 4).  decode steps 10, tokens 11 + 7 = 18.
    r = _hand_case([[3, 1, 2, 5], [1, 1, 4, 1], [2, 2, 1, 1]], P=3, B=2, N=9)
    assert list(r.status) == [oc.ABANDONED, oc.ABANDONED, oc.UNDRAWN]
    assert list(r.n) == [4, 4, 0] and list(r.s) == [0, 0, 0]
    assert list(r.decided_step) == [9, 5, -1] and list(r.decided_event) == [4, 3, -1]
    assert r.counters == {"rollouts": 8, "gen_tokens": 18, "prefill_tokens": 0, "decode_steps": 10, "events": 5,
                          "committed": 0, "abandoned": 2, "incomplete": 0, "prompts_drawn": 2}


def test_hand_worked_priority_beats_stream_order_at_one_boundary():
    # q0 [1,1,2,9], q1 [3,3,9,9]; B = 2, N = 6.
    # step 0: draw q0 (probe ends step 0, used 2), q1 (ends step 2, used 4).
    # end of 0: q0 n=2 -> continue, funded (used 5): j=2 (L=2) runs steps 1..2 (had it started at
    #           step 0 it would end at 1 and be funded alone).
    # end of 2: q0 n=3 (p_eff 0.2) and q1 n=2 (p_eff 0.4) decided together; one rollout of budget
    #           left: q1 first by p_eff (against stream order), j=2 (L=9) runs 3..11 (used 6);
    #           q0 cannot be funded -> INCOMPLETE.
    # end of 11: q1 n=3 -> continue, unfunded -> INCOMPLETE.  decode steps 12, tokens 4 + 15.
    r = _hand_case([[1, 1, 2, 9], [3, 3, 9, 9]], P=2, B=2, N=6)
    assert list(r.status) == [oc.INCOMPLETE, oc.INCOMPLETE]
    assert list(r.n) == [3, 3] and list(r.decided_step) == [-1, -1]
    assert r.counters == {"rollouts": 6, "gen_tokens": 19, "prefill_tokens": 0, "decode_steps": 12, "events": 3,
                          "committed": 0, "abandoned": 0, "incomplete": 2, "prompts_drawn": 2}
