"""The on-device controller (controller-only handle, no decode) against the Algorithm 1
oracle: every prompt's outcome, n, s and decision round, and every counter, bit-exact."""
import numpy as np
import pytest

import synth
from oracle import controller as oc

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def handle():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_26253_gb300 as pkg
    cfg = pkg.model_cfg(None, max_prompts=65536, max_active=8192, max_seqs=1, max_prompt_len=1, max_gen_len=1,
                        max_k=16)
    with pkg.Handle(cfg) as h:
        yield h


def _compare(h, w, si=None):
    si = si or synth.step_inputs(w)
    ref = oc.collect_workload(w, si)
    out = h.collect_step(thresholds=si.thresholds, lengths=si.lengths, N=w.budget_N, k=w.k, n0=w.n0, tau=w.tau,
                         target_B=w.target_B, reward_seed=w.reward_seed, prompt_len=w.prompt_len,
                         commit_min=w.commit_floor, prior=w.prior)
    assert np.array_equal(out.status, ref.status)
    assert np.array_equal(out.n, ref.n)
    assert np.array_equal(out.s, ref.s)
    assert np.array_equal(out.decided_round, ref.decided_round)
    for key, v in ref.counters.items():
        assert out.counters[key] == v, (key, out.counters[key], v)
    return out


@pytest.mark.parametrize("k", synth.SWEEP_K)
@pytest.mark.parametrize("n0", synth.SWEEP_N0)
def test_sweep_grid_bit_exact(handle, k, n0):
    for tau in synth.SWEEP_TAU:
        for rep in range(3):
            _compare(handle, synth.sweep_workload(k, n0, tau, rep))


def test_budget_binding_priority_and_edge_cases(handle):
    rng = np.random.default_rng(7)
    for it in range(60):
        k = int(rng.integers(2, 17))
        n0 = int(rng.integers(1, k + 1))
        P = int(rng.integers(1, 3000))
        B = int(rng.integers(1, min(P, 8192) + 1))
        w = synth.Workload("edge", None, n_prompts=P, prompt_len=int(rng.integers(1, 5)), target_B=B, k=k, n0=n0,
                           tau=float(rng.choice([0.0, 0.3, 0.45, 0.6, 1.0])), budget_N=int(rng.integers(0, 4 * P)),
                           commit_min=int(rng.integers(2, k + 1)),
                           prior=(int(rng.integers(1, 9)), int(rng.integers(1, 9))),
                           lengths=synth.Lengths("uniform", lo=1, hi=50),
                           seed_latent=it, seed_lengths=it + 1, reward_seed=it + 2)
        _compare(handle, w)


def test_working_set_equal_to_pool(handle):
    # B = P: the probe round spends the budget (B k > N) and no group reaches the commit floor
    w = synth.sweep_workload(8, 2, 0.45, 0, n_prompts=8192, target_B=8192)
    out = _compare(handle, w)
    assert out.counters["committed"] == 0


def test_ds_and_uniform_parameterisations(handle):
    # the comparison baselines as Algorithm 1 parameterisations (probe n0 = k, tau_low = 0;
    # uniform: a pool of B prompts with a budget of B k rollouts), bit-exact against the oracle
    from dataclasses import replace
    for k in (4, 8, 16):
        w = synth.sweep_workload(k, 2, 0.45, 5, n_prompts=8192, target_B=1024)
        _compare(handle, replace(w, n0=k, tau=0.0))
        _compare(handle, replace(w, n0=k, tau=0.0, n_prompts=1024, budget_N=1024 * k))


def test_length_difficulty_workload_sara_and_ds():
    # lengths tied to difficulty (all-fail prompts longest): token counts bit-exact for SARA and DS
    from dataclasses import replace
    import paper_2607_26253_gb300 as pkg
    cfg = pkg.model_cfg(None, max_prompts=8192, max_active=1024, max_seqs=1, max_prompt_len=1, max_gen_len=4096,
                        max_k=8)
    L = synth.Lengths("lognormal", median=1024, sigma=0.5, cap=4096, hard_scale=1.0)
    with pkg.Handle(cfg) as h:
        for rep in range(2):
            w = replace(synth.sweep_workload(8, 2, 0.45, rep, n_prompts=8192, target_B=1024), lengths=L)
            _compare(h, w)
            _compare(h, replace(w, n0=8, tau=0.0))


def _compare_async(h, w, si, schedule):
    from oracle import async_schedule as oa
    ref = oa.collect_workload(w, si, reserve=schedule == 2)
    out = h.collect_step(thresholds=si.thresholds, lengths=si.lengths, N=w.budget_N, k=w.k, n0=w.n0, tau=w.tau,
                         target_B=w.target_B, reward_seed=w.reward_seed, prompt_len=w.prompt_len,
                         commit_min=w.commit_floor, prior=w.prior, schedule=schedule)
    assert np.array_equal(out.status, ref.status)
    assert np.array_equal(out.n, ref.n) and np.array_equal(out.s, ref.s)
    assert np.array_equal(out.decided_round.astype(np.int32), np.minimum(ref.decided_event, 32767))
    c = ref.counters
    for key, v in (("rollouts", c["rollouts"]), ("gen_tokens", c["gen_tokens"]), ("decode_steps", c["decode_steps"]),
                   ("rounds", c["events"]), ("committed", c["committed"]), ("abandoned", c["abandoned"]),
                   ("incomplete", c["incomplete"]), ("prompts_drawn", c["prompts_drawn"]),
                   ("prefill_tokens", c["prefill_tokens"])):
        assert out.counters[key] == v, (key, out.counters[key], v)


def test_async_schedule_bit_exact():
    # the asynchronous per-prompt schedule (with and without the budget reservation) against
    # its oracle: random pools, then the 1.5B- and oversampled-shaped schedules
    import paper_2607_26253_gb300 as pkg
    cfg = pkg.model_cfg(None, max_prompts=2048, max_active=512, max_seqs=1, max_prompt_len=1, max_gen_len=8192,
                        max_k=16)
    rng = np.random.default_rng(21)
    with pkg.Handle(cfg) as h:
        for it in range(30):
            k = int(rng.integers(2, 17))
            n0 = int(rng.integers(1, k + 1))
            P = int(rng.integers(1, 2049))
            B = int(rng.integers(1, min(P, 512) + 1))
            w = synth.Workload("async", None, n_prompts=P, prompt_len=int(rng.integers(1, 5)), target_B=B, k=k,
                               n0=n0, tau=float(rng.choice([0.0, 0.3, 0.45, 0.6, 1.0])),
                               budget_N=int(rng.integers(0, 2 * P * k + 1)), commit_min=int(rng.integers(2, k + 1)),
                               prior=(int(rng.integers(1, 9)), int(rng.integers(1, 9))),
                               lengths=synth.Lengths("uniform", lo=1, hi=60), seed_latent=it,
                               seed_lengths=it + 1, reward_seed=it + 2)
            si = synth.step_inputs(w)
            for schedule in (1, 2):
                _compare_async(h, w, si, schedule)
        for name in ("1.5b", "oversampled"):
            w = synth.WORKLOADS[name]
            si = synth.step_inputs(w)
            for schedule in (1, 2):
                _compare_async(h, w, si, schedule)
