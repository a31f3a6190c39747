"""The DS and uniform baselines of the paper's comparisons (Fig. 5c/5d, 6a) as parameterisations
of the same Algorithm 1 controller, pinned to their own definitions:

- DS (dynamic sampling): draw prompts in stream order, generate all k rollouts of each at once,
  keep the groups whose rewards are mixed (0 < s < k), discard the rest, until B groups are kept.
  Here: probe n0 = k with tau_low = 0; a group decided at n = k is committed iff mixed (commit
  floor k) and abandoned iff all-same (the lossless limit of Thm. 1).
- uniform: the same on a pool of exactly B prompts with a budget of B k rollouts (each prompt
  gets k rollouts, no refill).

The expected yield of DS has a closed form over the synthetic difficulty mixture, and SARA's
rollout count against DS's on the same stream is the comparison the paper reports.
"""
from dataclasses import replace
from fractions import Fraction

import numpy as np

import synth
from oracle import controller as oc


def _beta_int(x: int, y: int) -> Fraction:
    # B(x, y) for positive integers: (x-1)! (y-1)! / (x+y-1)!
    from math import factorial
    return Fraction(factorial(x - 1) * factorial(y - 1), factorial(x + y - 1))


def _p_mixed(k: int, mixture) -> float:
    """P(a group of k rewards is mixed) when p = 0 w.p. m0, 1 w.p. m1, else Beta(2, 2):
    1 - E[p^k] - E[(1-p)^k], E[p^k] = B(2+k, 2) / B(2, 2) for the Beta(2, 2) part."""
    m0, m1, mb = mixture
    ek = _beta_int(2 + k, 2) / _beta_int(2, 2)
    return float(mb * (1 - 2 * ek))


def _ds(w: synth.Workload) -> synth.Workload:
    return replace(w, n0=w.k, tau=0.0, commit_min=None)


def test_ds_decides_every_prompt_in_its_probe_round_by_the_mixed_filter():
    w = _ds(synth.sweep_workload(8, 2, 0.45, 0, n_prompts=4096, target_B=512))
    si = synth.step_inputs(w)
    r = oc.collect_workload(w, si)
    drawn = r.counters["prompts_drawn"]
    v = oc.verdicts(si.thresholds, w.k, w.reward_seed)  # [P][k] 0/1 rewards, independent of the schedule
    s_all = v[:drawn].sum(axis=1)
    mixed = (s_all > 0) & (s_all < w.k)
    assert np.all(r.n[:drawn] == w.k)
    assert np.array_equal(r.s[:drawn], s_all)
    assert np.array_equal(r.status[:drawn] == oc.COMMITTED, mixed)
    assert np.array_equal(r.status[:drawn] == oc.ABANDONED, ~mixed)
    # every round draws at most B - |C| prompts and decides all of them: |C| reaches B exactly
    assert r.counters["committed"] == w.target_B
    assert r.counters["rollouts"] == w.k * drawn
    # a prompt is decided in the round that drew it: rounds = distinct decision rounds
    assert len(np.unique(r.decided_round[:drawn])) == r.counters["rounds"]


def test_uniform_is_ds_on_a_pool_of_B():
    B = 1024
    w = replace(_ds(synth.sweep_workload(8, 2, 0.45, 3, n_prompts=B, target_B=B)), budget_N=8 * B)
    si = synth.step_inputs(w)
    r = oc.collect_workload(w, si)
    v = oc.verdicts(si.thresholds, w.k, w.reward_seed)
    s_all = v.sum(axis=1)
    assert r.counters["prompts_drawn"] == B and r.counters["rounds"] == 1
    assert r.counters["rollouts"] == w.k * B
    assert r.counters["committed"] == int(((s_all > 0) & (s_all < w.k)).sum())


def test_ds_yield_matches_the_mixture_closed_form():
    # kept fraction of drawn prompts -> P(mixed); binomial tolerance (4 sigma) over ~17k draws
    k = 8
    w = _ds(synth.sweep_workload(k, 2, 0.45, 1, n_prompts=65536, target_B=6000))
    r = oc.collect_workload(w)
    drawn = r.counters["prompts_drawn"]
    pm = _p_mixed(k, w.mixture)
    frac = r.counters["committed"] / drawn
    assert abs(frac - pm) < 4 * np.sqrt(pm * (1 - pm) / drawn), (frac, pm, drawn)
    assert abs(pm - 0.4 * (1 - 2 * 6 / 110)) < 1e-12  # B(10,2)/B(2,2) = 6/110 at k = 8


def test_sara_spends_fewer_rollouts_than_ds_for_the_same_target():
    # the paper's comparison (Fig. 5c/5d): rollouts to reach B effective groups on one stream
    saved = []
    for rep in range(4):
        w = synth.sweep_workload(8, 2, 0.45, rep, n_prompts=8192, target_B=1024)
        sara = oc.collect_workload(w).counters
        ds = oc.collect_workload(_ds(w)).counters
        assert sara["committed"] >= w.target_B and ds["committed"] >= w.target_B
        saved.append(1 - sara["rollouts"] / ds["rollouts"])
    assert min(saved) > 0.12, saved


def test_hard_prompts_run_longest_in_the_length_generator():
    # median * (1 + hard_scale (1 - p)): all-fail prompts (p = 0) twice the all-pass median at
    # hard_scale = 1, so their mean lengths (same sigma, no cap in reach) are in ratio 2
    w = replace(synth.sweep_workload(8, 2, 0.45, 0, n_prompts=8192, target_B=1024),
                lengths=synth.Lengths("lognormal", median=1024, sigma=0.5, cap=10 ** 7, hard_scale=1.0))
    si = synth.step_inputs(w)
    p = si.thresholds.astype(np.float64) / 2.0 ** 32
    Lm = si.lengths.astype(np.float64).mean(axis=1)
    ratio = Lm[p == 0].mean() / Lm[p >= 1].mean()
    assert abs(ratio - 2.0) < 0.05, ratio
    base = synth.step_inputs(replace(w, lengths=replace(w.lengths, hard_scale=0.0)))
    assert abs(base.lengths[p == 0].mean() / base.lengths[p >= 1].mean() - 1.0) < 0.05


def test_token_savings_exceed_rollout_savings_when_hard_prompts_run_longest():
    # abandoned all-fail groups are the longest, so cutting them after the probe saves a larger
    # share of tokens than of rollouts (the paper's Fig. 6 observation)
    L = synth.Lengths("lognormal", median=1024, sigma=0.5, cap=4096, hard_scale=1.0)
    tot = np.zeros(4)
    for rep in range(4):
        w = replace(synth.sweep_workload(8, 2, 0.45, rep, n_prompts=8192, target_B=1024), lengths=L)
        sara = oc.collect_workload(w).counters
        ds = oc.collect_workload(_ds(w)).counters
        tot += [sara["rollouts"], ds["rollouts"], sara["gen_tokens"], ds["gen_tokens"]]
    roll_saving, tok_saving = 1 - tot[0] / tot[1], 1 - tot[2] / tot[3]
    assert roll_saving > 0.15 and tok_saving > roll_saving, (roll_saving, tok_saving)
