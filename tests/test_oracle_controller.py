"""Pins of the controller oracle O1 against what the paper and the mathematics fix.

Nothing here compares the oracle with itself: p_eff is checked against brute-force
Beta-Binomial enumeration and the closed form of Prop. 1, decisions against the
abandonment time of Thm. 2's proof, whole single-prompt runs against exact
expectations over every verdict pattern (Eq. EN and its commit-floor variant),
multi-prompt runs against Algorithm 1's invariants, and the seeded workloads against
the mixture's closed forms and Thms. 1 and 3 by Monte Carlo.
"""
import math
import os
from fractions import Fraction
from itertools import product

import numpy as np
import pytest

import synth
from oracle import controller as oc

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------------------- helpers
def beta_int(x: int, y: int) -> Fraction:
    """B(x, y) for positive integers: (x-1)!(y-1)!/(x+y-1)!."""
    return Fraction(math.factorial(x - 1) * math.factorial(y - 1), math.factorial(x + y - 1))


def peff_enumerated(n, s, k, a0, b0) -> Fraction:
    """P(1 <= S_k <= k-1 | n, s) by summing the Beta-Binomial predictive over every count m
    of successes among the r = k - n remaining rollouts (Beta identity of App. A)."""
    a, b = a0 + s, b0 + n - s
    r = k - n
    tot = Fraction(0)
    for m in range(r + 1):
        if 1 <= s + m <= k - 1:
            tot += math.comb(r, m) * beta_int(a + m, b + r - m) / beta_int(a, b)
    return tot


def first_abandon_n(k, tau, a0=1, b0=1):
    return next(n for n in range(1, k + 1) if oc.decide(n, 0, k, tau, alpha0=a0, beta0=b0) == oc.ABANDON)


PRIORS = [(1, 1), (2, 3), (3, 1), (1, 5), (8, 8), (4, 7)]


# ---------------------------------------------------------------------------- generator
def test_splitmix64_published_outputs():
    # SplitMix64 seeded with 0: first two outputs as published with the generator.
    assert synth.splitmix64_at(0, 1) == 0xE220A8397B1DCDAF
    assert synth.splitmix64_at(0, 2) == 0x6E789E6AA1B965F4


def test_oracle_verdict_hash_is_splitmix64():
    seed = 12345
    for q, j in [(0, 0), (3, 5), (70000, 63)]:
        h = synth.splitmix64_at(seed, q * 64 + j + 1) >> 32
        P = q + 1
        thr = np.zeros(P, np.uint64)
        thr[q] = h          # verdict = (h < thr) -> 0
        assert oc.verdicts(thr, 64, seed)[q, j] == 0
        thr[q] = h + 1      # -> 1
        assert oc.verdicts(thr, 64, seed)[q, j] == 1
    thr = np.array([0, 1 << 32], np.uint64)
    v = oc.verdicts(thr, 16, 7)
    assert v[0].sum() == 0 and v[1].sum() == 16


def test_verdict_rate_matches_threshold():
    thr = synth.constant_thresholds(20000, 0.3)
    v = oc.verdicts(thr, 8, 99)
    p = v.mean()
    assert abs(p - 0.3) < 4 * math.sqrt(0.3 * 0.7 / v.size)


# ---------------------------------------------------------------------------- p_eff (Prop. 1)
@pytest.mark.parametrize("a0,b0", PRIORS)
def test_peff_equals_beta_binomial_enumeration(a0, b0):
    for k in range(2, 13):
        for n in range(0, k + 1):
            for s in range(0, n + 1):
                assert oc.peff(n, s, k, a0, b0) == peff_enumerated(n, s, k, a0, b0), (k, n, s)


@pytest.mark.parametrize("k", [2, 4, 8, 16, 64])
def test_peff_uniform_prior_closed_form(k):
    # Prop. 1: with alpha0 = beta0 = 1, p_eff(n, 0) = p_eff(n, n) = (k - n)/(k + 1).
    for n in range(1, k + 1):
        assert oc.peff(n, 0, k) == Fraction(k - n, k + 1)
        assert oc.peff(n, n, k) == Fraction(k - n, k + 1)


@pytest.mark.parametrize("k", [4, 8, 16])
def test_peff_at_n0_keeps_both_saturated_completions(k):
    # Before any rollout both all-fail and all-pass completions are possible; the printed
    # formula's s = 0 branch (1 - B(a0, b0+k)/B(a0, b0) = k/(k+1) under Beta(1,1)) misses
    # the all-pass term.  Enumeration gives (k-1)/(k+1).
    assert oc.peff(0, 0, k) == Fraction(k - 1, k + 1)
    printed = 1 - beta_int(1, 1 + k) / beta_int(1, 1)
    assert printed == Fraction(k, k + 1) != oc.peff(0, 0, k)


@pytest.mark.parametrize("a0,b0", PRIORS)
def test_peff_monotone_and_mixed_absorbing(a0, b0):
    # Prop. 2: strictly decreasing along all-fail and all-pass prefixes; mixed => 1.
    for k in (4, 8, 16):
        fail = [oc.peff(n, 0, k, a0, b0) for n in range(1, k + 1)]
        ok = [oc.peff(n, n, k, a0, b0) for n in range(1, k + 1)]
        assert all(x > y for x, y in zip(fail, fail[1:]))
        assert all(x > y for x, y in zip(ok, ok[1:]))
        assert fail[-1] == 0 and ok[-1] == 0
        for n in range(2, k + 1):
            for s in range(1, n):
                assert oc.peff(n, s, k, a0, b0) == 1


# ---------------------------------------------------------------------------- DECIDE (Eq. decide)
@pytest.mark.parametrize("k", [4, 8, 16])
@pytest.mark.parametrize("tau", synth.SWEEP_TAU)
def test_first_abandon_matches_thm2_abandonment_time(k, tau):
    # Proof of Thm. 2: n_a = k - floor(tau (k+1)) under the uniform prior.  Eq. (decide)
    # abandons on the strict p_eff < tau, so when tau (k+1) is an integer the tie
    # p_eff(n_a) = tau continues one more rollout.
    t = Fraction(repr(tau))
    x = t * (k + 1)
    n_a = k - math.floor(x) + (1 if x.denominator == 1 else 0)
    assert first_abandon_n(k, tau) == min(n_a, k)


def test_first_abandon_golden_table():
    # tests/golden/first_abandon_n.txt: strict-rule abandonment rollout counts.
    rows = {}
    with open(os.path.join(GOLDEN, "first_abandon_n.txt")) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            k, *vals = line.split()
            rows[int(k)] = [int(v) for v in vals]
    for k, vals in rows.items():
        assert [first_abandon_n(k, t) for t in synth.SWEEP_TAU] == vals


def test_decide_commit_floor_and_lossless_limit():
    k = 8
    for n in range(2, k + 1):
        for s in range(1, n):
            for cm in (2, 4, 8):
                want = oc.COMMIT if n >= cm else oc.CONTINUE
                assert oc.decide(n, s, k, 0.45, commit_min=cm) == want
    # tau -> 0: only complete saturated groups are abandoned (Thm. 1, lossless limit).
    for n in range(1, k):
        assert oc.decide(n, 0, k, 0.0) == oc.CONTINUE
        assert oc.decide(n, n, k, 0.0) == oc.CONTINUE
    assert oc.decide(k, 0, k, 0.0) == oc.ABANDON
    assert oc.decide(k, k, k, 0.0) == oc.ABANDON
    # tau = 1: every all-same prefix is abandoned at the first decision.
    assert oc.decide(1, 0, k, 1.0) == oc.ABANDON


# ---------------------------------------------------------------------------- exact expectations
def _single_prompt_expectation(k, n0, tau, commit_min, gamma):
    """E[rollouts], P(commit) for one prompt by enumerating all 2^k verdict patterns."""
    EN = Fraction(0)
    Pc = Fraction(0)
    for bits in product((0, 1), repeat=k):
        s = sum(bits)
        w = gamma ** s * (1 - gamma) ** (k - s)
        r = oc.collect_step(None, None, k=k, n0=n0, tau=tau, target_B=1, N=k, commit_min=commit_min,
                            verdict_table=np.array([bits], np.uint8))
        EN += w * int(r.n[0])
        Pc += w * int(r.status[0] == oc.COMMITTED)
        assert r.status[0] in (oc.COMMITTED, oc.ABANDONED)
    return EN, Pc


@pytest.mark.parametrize("k,n0,tau", [(4, 1, 0.45), (4, 2, 0.3), (6, 1, 0.6), (6, 2, 0.45),
                                      (6, 3, 0.3), (5, 1, 0.4)])
@pytest.mark.parametrize("gamma", [Fraction(1, 10), Fraction(37, 100), Fraction(1, 2)])
def test_expected_rollouts_closed_forms(k, n0, tau, gamma):
    na = max(n0, first_abandon_n(k, tau))
    same = lambda n: gamma ** n + (1 - gamma) ** n
    # commit floor k (App. D default): a group mixed by n_a' runs to k, else stops at n_a'.
    EN, Pc = _single_prompt_expectation(k, n0, tau, k, gamma)
    assert EN == k - (k - na) * same(na)
    assert Pc == 1 - same(na)
    # commit at first mix (commit_min = 2): E[N] = n0 + sum_{n=n0}^{n_a'-1} P(same after n);
    # at n0 = 1 this is Eq. (EN): 1 + sum_{n=1}^{n_a-1} (gamma^n + (1-gamma)^n).
    EN2, Pc2 = _single_prompt_expectation(k, n0, tau, 2, gamma)
    assert EN2 == n0 + sum(same(n) for n in range(n0, na))
    assert Pc2 == 1 - same(na)
    if n0 == 1:
        assert EN2 == 1 + sum(gamma ** n + (1 - gamma) ** n for n in range(1, na))


# ---------------------------------------------------------------------------- Algorithm 1
def _check_invariants(thr, L, vt, k, n0, tau, B, N, cm, r, seed):
    P = thr.size
    st, n, s = r.status, r.n.astype(int), r.s.astype(int)
    c = r.counters
    assert c["rollouts"] <= N
    assert c["rollouts"] == n.sum()
    drawn = c["prompts_drawn"]
    assert np.all(st[:drawn] != oc.UNDRAWN) and np.all(st[drawn:] == oc.UNDRAWN)  # stream order
    assert np.all(n[drawn:] == 0)
    assert c["committed"] + c["abandoned"] + c["incomplete"] == drawn
    assert c["committed"] == int((st == oc.COMMITTED).sum())
    assert np.all(n[:drawn] >= n0) and np.all(n <= k)
    gen = sum(int(L[q, :n[q]].sum()) for q in range(P))
    assert c["gen_tokens"] == gen
    for q in range(drawn):
        v = vt[q, :n[q]]
        assert s[q] == v.sum()
        mixed = 0 < s[q] < n[q]
        if st[q] == oc.COMMITTED:
            assert mixed and n[q] >= cm
            # committed at the first decision where mixed and n >= commit_min
            if n[q] > max(cm, n0):
                pv = vt[q, :n[q] - 1]
                assert pv.min() == pv.max() or n[q] - 1 < cm
        elif st[q] == oc.ABANDONED:
            assert not mixed
            assert n[q] == k or oc.peff(n[q], s[q], k) < oc.tau_fraction(tau)
            if n[q] > n0:  # the previous decision continued
                assert oc.decide(n[q] - 1, s[q] - v[-1], k, tau, cm) == oc.CONTINUE
        else:
            assert st[q] == oc.INCOMPLETE
    if c["incomplete"] > 0:
        # a prompt is left undecided only when the target is met or the budget binds
        assert c["committed"] >= B or c["rollouts"] + 1 > N or c["rollouts"] + n0 > N
    if c["committed"] > B:  # overshoot only from the final round
        last = st == oc.COMMITTED
        assert r.decided_round[last].max() == c["rounds"] - 1


def test_algorithm1_invariants_random():
    rng = np.random.default_rng(2024)
    for it in range(300):
        k = int(rng.integers(2, 9))
        n0 = int(rng.integers(1, k + 1))
        cm = int(rng.integers(2, k + 1))
        tau = float(rng.choice(synth.SWEEP_TAU + (0.0, 0.1, 0.9, 1.0)))
        P = int(rng.integers(1, 40))
        B = int(rng.integers(1, P + 2))
        N = int(rng.integers(0, P * k + 3))
        p = rng.choice([0.0, 1.0, 0.5, 0.2, 0.8], size=P)
        thr = np.array([synth.constant_thresholds(1, x)[0] for x in p], np.uint64)
        L = rng.integers(1, 50, size=(P, k)).astype(np.int32)
        seed = int(rng.integers(0, 1 << 62))
        r = oc.collect_step(thr, L, k=k, n0=n0, tau=tau, target_B=B, N=N, reward_seed=seed,
                            commit_min=cm, prompt_len=7)
        vt = oc.verdicts(thr, k, seed)
        _check_invariants(thr, L, vt, k, n0, tau, B, N, cm, r, seed)
        # the hashed verdicts and the same verdicts passed as a table give the same step
        r2 = oc.collect_step(thr, L, k=k, n0=n0, tau=tau, target_B=B, N=N, commit_min=cm,
                             prompt_len=7, verdict_table=vt)
        assert np.array_equal(r.status, r2.status) and r.counters == r2.counters


def test_round_structure_and_decode_steps():
    w = synth.WORKLOADS["1.5b"]
    si = synth.step_inputs(w)
    r = oc.collect_workload(w, si)
    # round 0 probes B prompts with n0 rollouts (Alg. 1, first line)
    assert r.issued_per_round[0] == w.target_B * w.n0
    assert r.counters["rounds"] == len(r.issued_per_round)
    assert r.counters["prefill_tokens"] == r.counters["prompts_drawn"] * (w.prompt_len - 1)
    assert r.counters["rollouts"] == w.budget_N  # the budget binds on this workload


def test_budget_zero_and_empty_pool():
    r = oc.collect_step(np.zeros(5, np.uint64), np.ones((5, 4), np.int32), k=4, n0=2, tau=0.45,
                        target_B=3, N=1)
    assert r.counters["rollouts"] == 0 and r.counters["rounds"] == 0
    assert np.all(r.status == oc.UNDRAWN)
    r = oc.collect_step(np.zeros(0, np.uint64), np.ones((0, 4), np.int32), k=4, n0=2, tau=0.45,
                        target_B=3, N=100)
    assert r.counters["rollouts"] == 0


def test_target_stops_step():
    # every prompt mixed at the probe and commit at first mix: the step ends as soon as B commit
    k, B = 4, 5
    vt = np.tile(np.array([[1, 0, 1, 0]], np.uint8), (50, 1))
    r = oc.collect_step(None, np.ones((50, k), np.int32), k=k, n0=2, tau=0.45, target_B=B,
                        N=10_000, commit_min=2, verdict_table=vt)
    assert r.counters["committed"] == B and r.counters["rounds"] == 1
    assert r.counters["prompts_drawn"] == B


def test_priority_when_budget_binds():
    # Budget for exactly one continuation: the mixed prompt (p_eff = 1) outranks the all-fail one
    # even though it comes later in the stream; the all-fail one is left INCOMPLETE.
    k = 8
    vt = np.array([[0] * 8, [1, 0] + [1] * 6], np.uint8)
    r = oc.collect_step(None, np.ones((2, k), np.int32), k=k, n0=2, tau=0.1, target_B=2, N=5,
                        verdict_table=vt)
    assert list(r.n) == [2, 3] and r.status[0] == oc.INCOMPLETE
    # equal p_eff: the earlier stream index wins
    vt = np.array([[0] * 8, [0] * 8], np.uint8)
    r = oc.collect_step(None, np.ones((2, k), np.int32), k=k, n0=2, tau=0.1, target_B=2, N=5,
                        verdict_table=vt)
    assert list(r.n) == [3, 2]


# ---------------------------------------------------------------------------- Monte Carlo
def _mixture_phi(k, mix):
    # E[1 - g^k - (1-g)^k] with g ~ mixture; E_Beta(2,2)[g^k] = 6/((k+2)(k+3)).
    return mix[2] * (1 - 2 * 6 / ((k + 2) * (k + 3)))


@pytest.mark.parametrize("mix,cost,pcommit", [((0.35, 0.25, 0.40), 36 / 7, 2 / 7),
                                              ((0.45, 0.30, 0.25), 33 / 7, 5 / 28)])
def test_mixture_cost_and_commit_rate(mix, cost, pcommit):
    # k=8, n0=2, tau=.45 (n_a = 4), commit floor k, ample budget: a prompt is committed iff mixed
    # within 4 rollouts, so P(commit) = mix_beta * (1 - 2 E[g^4]) and E[N] = 4 + 4 P(commit).
    P = 40000
    w = synth.Workload("mc", None, n_prompts=P, prompt_len=1, target_B=P, k=8, n0=2, tau=0.45,
                       budget_N=8 * P, mixture=mix, seed_latent=11, reward_seed=12)
    si = synth.step_inputs(w)
    r = oc.collect_workload(w, si)
    n = r.n.astype(float)
    com = (r.status == oc.COMMITTED).astype(float)
    assert abs(n.mean() - cost) < 4 * n.std() / math.sqrt(P)
    assert abs(com.mean() - pcommit) < 4 * math.sqrt(pcommit * (1 - pcommit) / P)
    # Phi of the mixture under uniform k-sampling (Def. 1)
    v = oc.verdicts(si.thresholds, 8, w.reward_seed)
    eff = ((v.sum(1) > 0) & (v.sum(1) < 8)).astype(float)
    phi = _mixture_phi(8, mix)
    assert abs(eff.mean() - phi) < 4 * math.sqrt(phi * (1 - phi) / P)


def test_thm1_abandonment_reliability_under_prior():
    # gamma ~ Beta(1,1): the fraction of abandoned prompts whose completed group would have been
    # effective equals E[p_eff at abandonment] (tower rule) and is < tau.
    P, k, tau = 60000, 8, 0.45
    rng = np.random.default_rng(5)
    thr = np.floor(rng.random(P) * 4294967296.0).astype(np.uint64)
    r = oc.collect_step(thr, np.ones((P, k), np.int32), k=k, n0=2, tau=tau, target_B=P, N=k * P,
                        reward_seed=77)
    ab = r.status == oc.ABANDONED
    v = oc.verdicts(thr, k, 77)[ab]
    lost = ((v.sum(1) > 0) & (v.sum(1) < k)).astype(float)
    pe = np.array([float(oc.peff(int(n), int(s), k)) for n, s in zip(r.n[ab], r.s[ab])])
    assert abs(lost.mean() - pe.mean()) < 4 * lost.std() / math.sqrt(lost.size)
    assert lost.mean() <= tau
    assert np.all(pe < tau)


def test_thm3_fixed_budget_yield_dominates_uniform():
    # Same budget N: SARA's committed groups exceed the mixed count of uniform allocation's N/k
    # full groups (expected Phi N / k).  The exchange argument of the proof ignores the groups
    # left INCOMPLETE when the budget runs out mid-group; those losses grow with the working set
    # (B - |C|), so the comparison runs with B = N/(2k), a target SARA does not reach, so it
    # spends the whole budget.  (A working set of B*n0 >= N commits nothing; tested below.)
    k, N = 8, 4096
    ys, yu = [], []
    for rep in range(12):
        w = synth.Workload("mc", None, n_prompts=4 * N, prompt_len=1, target_B=N // (2 * k), k=k, n0=2,
                           tau=0.45, budget_N=N, seed_latent=300 + rep, reward_seed=400 + rep)
        si = synth.step_inputs(w)
        r = oc.collect_workload(w, si)
        ys.append(r.counters["committed"])
        v = oc.verdicts(si.thresholds[: N // k], k, w.reward_seed)
        yu.append(int(((v.sum(1) > 0) & (v.sum(1) < k)).sum()))
    assert np.mean(ys) > np.mean(yu)
    assert np.mean(ys) > _mixture_phi(k, (0.35, 0.25, 0.40)) * N / k


def test_oversized_working_set_commits_nothing_at_commit_floor_k():
    # B * n0 >= N: the probe round alone spends the budget, no group reaches k rollouts.
    k, N = 8, 1024
    w = synth.Workload("edge", None, n_prompts=4 * N, prompt_len=1, target_B=N, k=k, n0=2,
                       tau=0.45, budget_N=N)
    r = oc.collect_workload(w)
    assert r.counters["committed"] == 0 and r.counters["rollouts"] == N


@pytest.mark.parametrize("gamma", [0.0, 0.1, 0.5, 0.9, 1.0])
def test_thm2_expected_rollouts_monte_carlo(gamma):
    P, k, n0, tau = 30000, 8, 2, 0.45
    thr = synth.constant_thresholds(P, gamma)
    r = oc.collect_step(thr, np.ones((P, k), np.int32), k=k, n0=n0, tau=tau, target_B=P, N=k * P,
                        reward_seed=31)
    g = float(thr[0]) / 4294967296.0
    na = max(n0, first_abandon_n(k, tau))
    want = k - (k - na) * (g ** na + (1 - g) ** na)
    n = r.n.astype(float)
    sd = max(n.std(), 1e-9)
    assert abs(n.mean() - want) < 4 * sd / math.sqrt(P) + 1e-12
