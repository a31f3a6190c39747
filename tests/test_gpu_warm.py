"""Warm-start on the GPU controller against the warm-start oracle (oracle/warm_start.py).

Several steps over the same recurring prompts, each step starting from the priors the oracle
carried out of the previous one (decay 0.9): every prompt's outcome, n, s and decision round and
the step counters must equal the oracle's, including the steps where the budget binds (continuing
prompts ranked by their fp64 p_eff).  The predictor is fp64 on both sides (log-Gamma), so the
cases are checked to sit away from ties first.  The carried priors the library returns must
equal the oracle's carry bit for bit."""
import math

import numpy as np
import pytest

import synth
from gpu_util import handle_cfg
from oracle import async_schedule as oa
from oracle import controller as oc
from oracle import warm_start as ow

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def pkg():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_26253_gb300 as p
    p.load()
    return p


def _min_margin(si, a, b, w, r):
    """Smallest |p_eff - tau| over every (n, s) a drawn prompt of the oracle's run reached."""
    m = math.inf
    for q in np.nonzero(r.n)[0]:
        for nn in range(w.n0, int(r.n[q]) + 1):
            v = oc.verdicts(si.thresholds[q:q + 1], w.k, w.reward_seed)[0]
            ss = int(v[:nn].sum())
            if ss in (0, nn) and nn < w.k:
                m = min(m, abs(ow.peff(nn, ss, w.k, float(a[q]), float(b[q])) - w.tau))
    return m


@pytest.mark.parametrize("budget_factor", [8, 3])  # 3: the budget binds, continuing prompts are ranked
def test_warm_start_steps_match_the_oracle(pkg, budget_factor):
    P, B, steps, lam = 2048, 192, 5, 0.9
    w0 = synth.Workload("warm", None, n_prompts=P, prompt_len=1, target_B=B, k=8, n0=2, tau=0.45,
                        budget_N=budget_factor * B * 2, lengths=synth.Lengths("uniform", lo=1, hi=9))
    cfg = pkg.model_cfg(None, max_prompts=P, max_active=B, max_seqs=1, max_prompt_len=1, max_gen_len=16, max_k=8)
    si = synth.step_inputs(w0)
    a, b = np.ones(P), np.ones(P)
    with pkg.Handle(cfg) as h:
        for t in range(steps):
            w = synth.Workload(w0.name, None, n_prompts=P, prompt_len=1, target_B=B, k=8, n0=2, tau=0.45,
                               budget_N=w0.budget_N, lengths=w0.lengths, reward_seed=100 + t)
            ref = ow.collect_step(si.thresholds, si.lengths, a, b, k=8, n0=2, tau=0.45, target_B=B, N=w.budget_N,
                                  reward_seed=w.reward_seed)
            assert _min_margin(si, a, b, w, ref) > 1e-9
            out = h.collect_step(thresholds=si.thresholds, lengths=si.lengths, N=w.budget_N, k=8, n0=2, tau=0.45,
                                 target_B=B, reward_seed=w.reward_seed, prior_a=a, prior_b=b, decay=lam,
                                 want_next_prior=True)
            assert np.array_equal(out.status, ref.status), t
            assert np.array_equal(out.n, ref.n) and np.array_equal(out.s, ref.s), t
            assert np.array_equal(out.decided_round, ref.decided_round), t
            for key in ("rollouts", "gen_tokens", "rounds", "committed", "abandoned", "incomplete", "prompts_drawn"):
                assert out.counters[key] == ref.counters[key], (t, key)
            a, b = ow.carry(a, b, ref.n, ref.s, 1.0, 1.0, lam)
            assert np.array_equal(out.prior_next[0], a) and np.array_equal(out.prior_next[1], b), t


def test_warm_start_on_the_decode_engine(pkg):
    """The tiny policy: a step with carried priors decodes every issued rollout and its schedule
    equals the oracle's."""
    w = synth.WORKLOADS["tiny"]
    weights = synth.model_weights(w.model, w.weight_seed)
    si = synth.step_inputs(w)
    rng = np.random.default_rng(4)
    a = 1.0 + 0.9 * rng.integers(0, 5, w.n_prompts)  # as if carried from earlier steps
    b = 1.0 + 0.9 * rng.integers(0, 5, w.n_prompts)
    ref = ow.collect_step(si.thresholds, si.lengths, a, b, k=w.k, n0=w.n0, tau=w.tau, target_B=w.target_B,
                          N=w.budget_N, reward_seed=w.reward_seed, prompt_len=w.prompt_len)
    assert _min_margin(si, a, b, w, ref) > 1e-9
    with pkg.Handle(handle_cfg(w, pkg), weights) as h:
        out = h.collect_step(thresholds=si.thresholds, lengths=si.lengths, tokens=si.tokens, N=w.budget_N, k=w.k,
                             n0=w.n0, tau=w.tau, target_B=w.target_B, reward_seed=w.reward_seed,
                             sample_seed=w.sample_seed, prior_a=a, prior_b=b)
    assert np.array_equal(out.status, ref.status) and np.array_equal(out.n, ref.n)
    assert np.array_equal(out.decided_round, ref.decided_round)
    for key, v in ref.counters.items():
        assert out.counters[key] == v, key


def test_warm_start_arguments_rejected(pkg):
    w = synth.sweep_workload(8, 2, 0.45, n_prompts=64, target_B=16)
    si = synth.step_inputs(w)
    cfg = pkg.model_cfg(None, max_prompts=64, max_active=16, max_seqs=1, max_prompt_len=1, max_gen_len=1, max_k=8)
    with pkg.Handle(cfg) as h:
        kw = dict(thresholds=si.thresholds, lengths=si.lengths, N=w.budget_N, k=8, n0=2, tau=0.45, target_B=16,
                  reward_seed=1)
        for bad in ({"prior_a": np.ones(64)}, {"prior_a": np.ones(64), "prior_b": np.zeros(64)},
                    {"decay": 1.5}, {"prior_a": np.ones(64), "prior_b": np.full(64, np.inf)}):
            with pytest.raises(pkg.SaraError) as e:
                h.collect_step(**kw, **bad)
            assert e.value.code == pkg.SARA_EINVAL


@pytest.mark.parametrize("schedule", [1, 2])
def test_warm_start_with_the_asynchronous_schedule(pkg, schedule):
    """Controller-only handle, several steps with carried priors on the asynchronous schedule
    (2: with the budget reserve); the budget binds, so continuing prompts at one boundary are
    ranked by their fp64 p_eff.  Every prompt's outcome, n, s and deciding event, the counters
    and the carried priors equal the oracle's."""
    P, B, steps, lam = 1024, 96, 4, 0.9
    base = synth.Workload("warm-async", None, n_prompts=P, prompt_len=1, target_B=B, k=8, n0=2, tau=0.45,
                          budget_N=3 * B * 2, lengths=synth.Lengths("uniform", lo=1, hi=40))
    cfg = pkg.model_cfg(None, max_prompts=P, max_active=B, max_seqs=1, max_prompt_len=1, max_gen_len=64, max_k=8)
    si = synth.step_inputs(base)
    a, b = np.ones(P), np.ones(P)
    with pkg.Handle(cfg) as h:
        for t in range(steps):
            seed = 300 + t
            ref = oa.collect_step(si.thresholds, si.lengths, k=8, n0=2, tau=0.45, target_B=B, N=base.budget_N,
                                  reward_seed=seed, reserve=schedule == 2, prior_a=a, prior_b=b)
            w = synth.Workload(base.name, None, n_prompts=P, prompt_len=1, target_B=B, k=8, n0=2, tau=0.45,
                               budget_N=base.budget_N, lengths=base.lengths, reward_seed=seed)
            assert _min_margin(si, a, b, w, ref) > 1e-9
            out = h.collect_step(thresholds=si.thresholds, lengths=si.lengths, N=base.budget_N, k=8, n0=2, tau=0.45,
                                 target_B=B, reward_seed=seed, prior_a=a, prior_b=b, decay=lam,
                                 want_next_prior=True, schedule=schedule)
            assert np.array_equal(out.status, ref.status), t
            assert np.array_equal(out.n, ref.n) and np.array_equal(out.s, ref.s), t
            assert np.array_equal(out.decided_round.astype(np.int32), np.minimum(ref.decided_event, 32767)), t
            c = ref.counters
            for key, v in (("rollouts", c["rollouts"]), ("gen_tokens", c["gen_tokens"]),
                           ("decode_steps", c["decode_steps"]), ("rounds", c["events"]),
                           ("committed", c["committed"]), ("incomplete", c["incomplete"])):
                assert out.counters[key] == v, (t, key)
            a, b = ow.carry(a, b, ref.n, ref.s, 1.0, 1.0, lam)
            assert np.array_equal(out.prior_next[0], a) and np.array_equal(out.prior_next[1], b), t


def test_warm_start_with_the_asynchronous_schedule_on_the_decode_engine(pkg):
    """The tiny policy on the asynchronous schedule with carried priors: decisions at every
    decode-step boundary take each prompt's own prior; the schedule equals the oracle's."""
    w = synth.WORKLOADS["tiny"]
    weights = synth.model_weights(w.model, w.weight_seed)
    si = synth.step_inputs(w)
    rng = np.random.default_rng(5)
    a = 1.0 + 0.9 * rng.integers(0, 5, w.n_prompts)
    b = 1.0 + 0.9 * rng.integers(0, 5, w.n_prompts)
    ref = oa.collect_step(si.thresholds, si.lengths, k=w.k, n0=w.n0, tau=w.tau, target_B=w.target_B, N=w.budget_N,
                          reward_seed=w.reward_seed, prompt_len=w.prompt_len, prior_a=a, prior_b=b)
    assert _min_margin(si, a, b, w, ref) > 1e-9
    with pkg.Handle(handle_cfg(w, pkg), weights) as h:
        out = h.collect_step(thresholds=si.thresholds, lengths=si.lengths, tokens=si.tokens, N=w.budget_N, k=w.k,
                             n0=w.n0, tau=w.tau, target_B=w.target_B, reward_seed=w.reward_seed,
                             sample_seed=w.sample_seed, prior_a=a, prior_b=b, schedule=1)
    assert np.array_equal(out.status, ref.status) and np.array_equal(out.n, ref.n)
    assert np.array_equal(out.decided_round.astype(np.int32), np.minimum(ref.decided_event, 32767))
    assert out.counters["decode_steps"] == ref.counters["decode_steps"]
    assert out.counters["gen_tokens"] == ref.counters["gen_tokens"]
