"""Pins of the warm-start oracle (oracle/warm_start.py): the real-prior predictor against the
product form of the Beta-function ratios and against O1's exact rationals, the step against O1
when every prior is the integer base prior, the carry rule's limits, the paper's statement that a
prompt seen saturated starts skewed and is abandoned after fewer probes, and its effect on a
stream of recurring prompts over several steps."""
from fractions import Fraction

import numpy as np
import pytest

import synth
from oracle import controller as oc
from oracle import warm_start as ow


def _ratio_product(a: float, b: float, r: int) -> float:
    """B(a, b + r) / B(a, b) = prod_{i<r} (b + i) / (a + b + i) for an integer r >= 0."""
    out = 1.0
    for i in range(r):
        out *= (b + i) / (a + b + i)
    return out


def test_real_prior_peff_matches_the_product_form():
    rng = np.random.default_rng(3)
    for _ in range(400):
        k = int(rng.integers(2, 17))
        n = int(rng.integers(1, k))
        a, b = float(rng.uniform(0.3, 12.0)), float(rng.uniform(0.3, 12.0))
        r = k - n
        # s = 0: the completion is all-fail with prob B(a, b + n + r) / B(a, b + n)
        want0 = 1.0 - _ratio_product(a, b + n, r)
        # s = n: all-pass with prob B(a + n + r, b) / B(a + n, b) (the mirror: swap a and b)
        wantn = 1.0 - _ratio_product(b, a + n, r)
        assert abs(ow.peff(n, 0, k, a, b) - want0) < 1e-12
        assert abs(ow.peff(n, n, k, a, b) - wantn) < 1e-12
        if n >= 2:
            assert ow.peff(n, 1, k, a, b) == 1.0


def test_integer_priors_reproduce_the_exact_predictor():
    for k in (4, 8, 16):
        for a0, b0 in ((1, 1), (2, 3), (5, 1)):
            for n in range(1, k + 1):
                for s in range(0, n + 1):
                    exact = oc.peff(n, s, k, a0, b0)
                    assert abs(ow.peff(n, s, k, float(a0), float(b0)) - float(exact)) < 1e-14


def _tie_free(k, tau, a0, b0, margin=Fraction(1, 10 ** 9)):
    t = oc.tau_fraction(tau)
    return all(abs(oc.peff(n, s, k, a0, b0) - t) > margin for n in range(1, k + 1) for s in (0, n))


def test_uniform_integer_priors_reproduce_the_round_synchronous_oracle():
    rng = np.random.default_rng(5)
    checked = 0
    for it in range(60):
        k = int(rng.choice([4, 8, 16]))
        tau = float(rng.choice([0.3, 0.45, 0.55]))
        a0, b0 = int(rng.integers(1, 4)), int(rng.integers(1, 4))
        if not _tie_free(k, tau, a0, b0):
            continue
        n0 = int(rng.integers(1, k + 1))
        P = int(rng.integers(1, 300))
        w = synth.Workload("warm", None, n_prompts=P, prompt_len=1, target_B=int(rng.integers(1, P + 1)), k=k, n0=n0,
                           tau=tau, budget_N=int(rng.integers(0, 3 * P * k // 2 + 1)),
                           commit_min=int(rng.integers(2, k + 1)), prior=(a0, b0),
                           lengths=synth.Lengths("uniform", lo=1, hi=40), seed_latent=it, seed_lengths=it + 1,
                           reward_seed=it + 2)
        si = synth.step_inputs(w)
        ref = oc.collect_workload(w, si)
        got = ow.collect_step(si.thresholds, si.lengths, np.full(P, float(a0)), np.full(P, float(b0)), k=k, n0=n0,
                              tau=tau, target_B=w.target_B, N=w.budget_N, reward_seed=w.reward_seed,
                              commit_min=w.commit_floor, prompt_len=1)
        assert np.array_equal(got.status, ref.status) and np.array_equal(got.n, ref.n)
        assert np.array_equal(got.s, ref.s) and np.array_equal(got.decided_round, ref.decided_round)
        assert got.counters == ref.counters
        checked += 1
    assert checked >= 30


def test_carry_limits_and_a_hand_worked_update():
    a = np.array([1.0, 2.5, 1.0])
    b = np.array([1.0, 1.0, 4.0])
    n = np.array([4, 0, 8])
    s = np.array([1, 0, 8])
    a0, b0 = ow.carry(a, b, n, s, 1.0, 1.0, 0.0)
    assert np.all(a0 == 1.0) and np.all(b0 == 1.0)            # lambda = 0: plain SARA every step
    a1, b1 = ow.carry(a, b, n, s, 1.0, 1.0, 1.0)
    assert list(a1) == [2.0, 2.5, 9.0] and list(b1) == [4.0, 1.0, 4.0]   # lambda = 1: counts add up
    ah, bh = ow.carry(a, b, n, s, 1.0, 1.0, 0.5)
    assert list(ah) == [1.5, 1.75, 5.0] and list(bh) == [2.5, 1.0, 2.5]  # 1 + 0.5 (a - 1 + s), ...


def test_a_prompt_seen_saturated_is_abandoned_after_fewer_probes():
    # k = 8, tau = 0.45, base prior Beta(1, 1).  Without history an all-fail probe of 2 gives
    # p_eff = (8 - 2) / 9 = 0.667: continue; the strict rule abandons at n = 4 (4/9 < 0.45).
    # After a step with 6 failures and lambda = 0.9 the prior is Beta(1, 1 + 5.4); with a = 1,
    # B(1, y + r) / B(1, y) = y / (y + r), so after the same probe p_eff = 1 - 8.4 / 14.4 = 0.417:
    # abandoned at the probe.
    k, tau = 8, 0.45
    assert ow.decide(2, 0, k, tau, k, 1.0, 1.0) == oc.CONTINUE
    assert ow.decide(4, 0, k, tau, k, 1.0, 1.0) == oc.ABANDON
    a, b = ow.carry(np.array([1.0]), np.array([1.0]), np.array([6]), np.array([0]), 1.0, 1.0, 0.9)
    assert abs(b[0] - 6.4) < 1e-12 and a[0] == 1.0
    assert abs(ow.peff(2, 0, k, float(a[0]), float(b[0])) - (1 - 8.4 / 14.4)) < 1e-12
    assert ow.decide(2, 0, k, tau, k, float(a[0]), float(b[0])) == oc.ABANDON


def _multi_step(lam, steps=6, P=3000, B=256):
    w = synth.Workload("warm", None, n_prompts=P, prompt_len=1, target_B=B, k=8, n0=2, tau=0.45,
                       budget_N=8 * P, lengths=synth.Lengths("uniform", lo=1, hi=1))
    si = synth.step_inputs(w)  # the same prompts (latent rates) every step, fresh verdicts per step
    a, b = np.ones(P), np.ones(P)
    rollouts = commits = 0
    for t in range(steps):
        r = ow.collect_step(si.thresholds, si.lengths, a, b, k=8, n0=2, tau=0.45, target_B=B, N=8 * P,
                            reward_seed=1000 + t)
        rollouts += r.counters["rollouts"]
        commits += r.counters["committed"]
        a, b = ow.carry(a, b, r.n, r.s, 1.0, 1.0, lam)
    return rollouts / commits


@pytest.mark.slow
def test_history_reduces_rollouts_per_effective_group_on_recurring_prompts():
    # a stream of recurring prompts (35 % never solved, 25 % always solved, 40 % Beta(2, 2)):
    # carrying the evidence lets saturated prompts be abandoned at the probe
    plain, warm = _multi_step(0.0), _multi_step(0.9)
    assert warm < 0.95 * plain, (plain, warm)


# ---- the warm-start on the asynchronous schedule (oracle/async_schedule.py with prior_a / prior_b)
from oracle import async_schedule as oa  # noqa: E402


def _async_case(rng, it, equal_len=None):
    k = int(rng.choice([4, 8, 16]))
    tau = float(rng.choice([0.3, 0.45, 0.55]))
    n0 = int(rng.integers(1, k + 1))
    P = int(rng.integers(1, 300))
    lengths = synth.Lengths("uniform", lo=1, hi=40) if equal_len is None else synth.Lengths("uniform", lo=equal_len,
                                                                                         hi=equal_len)
    return synth.Workload("warm-async", None, n_prompts=P, prompt_len=1, target_B=int(rng.integers(1, P + 1)), k=k,
                          n0=n0, tau=tau, budget_N=int(rng.integers(0, 3 * P * k // 2 + 1)),
                          commit_min=int(rng.integers(2, k + 1)), prior=(int(rng.integers(1, 4)), int(rng.integers(1, 4))),
                          lengths=lengths, seed_latent=it, seed_lengths=it + 1, reward_seed=it + 2)


@pytest.mark.parametrize("reserve", [False, True])
def test_async_with_uniform_integer_priors_is_the_integer_async_oracle(reserve):
    """Real priors all equal to the integer base prior: the float64 predictor takes the same
    decisions and the same priority order as the exact one (cases with a tie excluded)."""
    rng = np.random.default_rng(21)
    checked = 0
    for it in range(80):
        w = _async_case(rng, it)
        a0, b0 = w.prior
        if not _tie_free(w.k, w.tau, a0, b0):
            continue
        si = synth.step_inputs(w)
        kw = dict(k=w.k, n0=w.n0, tau=w.tau, target_B=w.target_B, N=w.budget_N, reward_seed=w.reward_seed,
                  commit_min=w.commit_floor, prior=w.prior, reserve=reserve)
        ref = oa.collect_step(si.thresholds, si.lengths, **kw)
        got = oa.collect_step(si.thresholds, si.lengths, prior_a=np.full(w.n_prompts, float(a0)),
                              prior_b=np.full(w.n_prompts, float(b0)), **kw)
        assert np.array_equal(got.status, ref.status) and np.array_equal(got.n, ref.n), it
        assert np.array_equal(got.s, ref.s) and np.array_equal(got.decided_step, ref.decided_step), it
        assert got.counters == ref.counters, it
        checked += 1
    assert checked >= 40


def test_async_with_real_priors_and_equal_lengths_is_the_round_synchronous_warm_oracle():
    """Every rollout the same length: each step boundary with decisions is a round, so the
    asynchronous schedule with per-prompt real priors equals O1w's round-synchronous step."""
    rng = np.random.default_rng(22)
    for it in range(60):
        Lc = int(rng.integers(1, 30))
        w = _async_case(rng, it, equal_len=Lc)
        si = synth.step_inputs(w)
        a = rng.uniform(0.5, 6.0, w.n_prompts)
        b = rng.uniform(0.5, 6.0, w.n_prompts)
        sync = ow.collect_step(si.thresholds, si.lengths, a, b, k=w.k, n0=w.n0, tau=w.tau, target_B=w.target_B,
                               N=w.budget_N, reward_seed=w.reward_seed, commit_min=w.commit_floor)
        asy = oa.collect_step(si.thresholds, si.lengths, k=w.k, n0=w.n0, tau=w.tau, target_B=w.target_B,
                              N=w.budget_N, reward_seed=w.reward_seed, commit_min=w.commit_floor, prior_a=a,
                              prior_b=b)
        assert np.array_equal(asy.status, sync.status), it
        assert np.array_equal(asy.n, sync.n) and np.array_equal(asy.s, sync.s), it
        assert np.array_equal(asy.decided_event, sync.decided_round.astype(np.int32)), it
        for key in ("rollouts", "gen_tokens", "committed", "abandoned", "incomplete", "prompts_drawn"):
            assert asy.counters[key] == sync.counters[key], (it, key)
        assert asy.counters["decode_steps"] == sync.counters["rounds"] * Lc


def test_async_warm_start_abandons_a_prompt_seen_saturated_at_its_probe():
    """The hand-worked case of the round schedule, on the asynchronous one: after a step of six
    failures with lambda = 0.9 the prior is Beta(1, 6.4) and the all-fail probe of 2 has p_eff =
    1 - 8.4 / 14.4 < 0.45, so the prompt is abandoned when its probe finishes; without the carried
    prior it continues."""
    thr = np.array([0], dtype=np.uint64)  # never solved
    lengths = np.array([[3, 5, 2, 4, 6, 1, 7, 2]], dtype=np.int64)
    kw = dict(k=8, n0=2, tau=0.45, target_B=1, N=16, reward_seed=0)
    plain = oa.collect_step(thr, lengths, **kw)
    warm = oa.collect_step(thr, lengths, prior_a=np.array([1.0]), prior_b=np.array([6.4]), **kw)
    assert warm.status[0] == oc.ABANDONED and warm.n[0] == 2 and warm.decided_step[0] == 4  # probe ends at step 4
    assert plain.status[0] == oc.ABANDONED and plain.n[0] == 4  # abandoned at n = 4 (4/9 < 0.45)
