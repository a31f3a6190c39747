"""The step's failure paths, made to fire without faulting or hanging the GPU.

Every device wait of the decode step is bounded.  sara_set_limits tightens the bounds for a
test: a phase counter whose waits can never complete (a value nothing reaches) must make the
call return SARA_ETIMEOUT within the wait limit, and a bound on the step loop's iterations
must end the loop with SARA_ETIMEOUT; in both cases the handle must stay usable, i.e. the next
call with the default limits reproduces the oracle's schedule bit-exactly.
"""
import time

import numpy as np
import pytest

import synth
from gpu_util import handle_cfg
from oracle import controller as oc

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def pkg():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_26253_gb300 as p
    p.load()
    return p


def _step(h, w, si):
    return h.collect_step(thresholds=si.thresholds, lengths=si.lengths, tokens=si.tokens, N=w.budget_N, k=w.k,
                          n0=w.n0, tau=w.tau, target_B=w.target_B, reward_seed=w.reward_seed,
                          sample_seed=w.sample_seed, commit_min=w.commit_floor, prior=w.prior)


def _assert_oracle_schedule(out, w, si):
    ref = oc.collect_workload(w, si)
    assert np.array_equal(out.status, ref.status)
    assert np.array_equal(out.n, ref.n) and np.array_equal(out.s, ref.s)
    for key, v in ref.counters.items():
        assert out.counters[key] == v, (key, out.counters[key], v)


@pytest.mark.parametrize("phase", [0, 1, 4, 11])  # embedding; QKV, O-projection of layer 0; FIN_Q of layer 1
def test_stalled_phase_times_out_and_handle_recovers(pkg, phase):
    w = synth.WORKLOADS["tiny"]
    weights = synth.model_weights(w.model, w.weight_seed)
    si = synth.step_inputs(w)
    with pkg.Handle(handle_cfg(w, pkg), weights) as h:
        h.set_limits(wait_limit_ns=20_000_000, stall_phase=phase)  # 20 ms
        t0 = time.time()
        with pytest.raises(pkg.SaraError) as e:
            _step(h, w, si)
        assert e.value.code == pkg.SARA_ETIMEOUT
        assert time.time() - t0 < 30.0
        h.set_limits()  # defaults again: the same handle runs the step exactly
        _assert_oracle_schedule(_step(h, w, si), w, si)


def test_loop_iteration_bound(pkg):
    w = synth.WORKLOADS["tiny"]
    weights = synth.model_weights(w.model, w.weight_seed)
    si = synth.step_inputs(w)
    with pkg.Handle(handle_cfg(w, pkg), weights) as h:
        h.set_limits(max_loop_iters=5)
        with pytest.raises(pkg.SaraError) as e:
            _step(h, w, si)
        assert e.value.code == pkg.SARA_ETIMEOUT
        h.set_limits()
        _assert_oracle_schedule(_step(h, w, si), w, si)


def test_loop_iteration_bound_controller_only(pkg):
    w = synth.sweep_workload(8, 2, 0.45, n_prompts=4096, target_B=512)
    si = synth.step_inputs(w)
    cfg = pkg.model_cfg(None, max_prompts=w.n_prompts, max_active=w.target_B, max_seqs=1, max_prompt_len=1,
                        max_gen_len=1, max_k=w.k)
    with pkg.Handle(cfg) as h:
        h.set_limits(max_loop_iters=3)
        with pytest.raises(pkg.SaraError) as e:
            h.collect_step(thresholds=si.thresholds, lengths=si.lengths, N=w.budget_N, k=w.k, n0=w.n0, tau=w.tau,
                           target_B=w.target_B, reward_seed=w.reward_seed)
        assert e.value.code == pkg.SARA_ETIMEOUT
        h.set_limits()
        out = h.collect_step(thresholds=si.thresholds, lengths=si.lengths, N=w.budget_N, k=w.k, n0=w.n0, tau=w.tau,
                             target_B=w.target_B, reward_seed=w.reward_seed)
        ref = oc.collect_workload(w, si)
        assert np.array_equal(out.status, ref.status) and out.counters["rollouts"] == ref.counters["rollouts"]


def test_limits_out_of_range_rejected(pkg):
    w = synth.WORKLOADS["tiny"]
    weights = synth.model_weights(w.model, w.weight_seed)
    with pkg.Handle(handle_cfg(w, pkg), weights) as h:
        for kw in ({"wait_limit_ns": -1}, {"max_loop_iters": -2}, {"stall_phase": -5}, {"stall_phase": 10 ** 6},
                   {"eager_softmax": 2}):
            with pytest.raises(pkg.SaraError) as e:
                h.set_limits(**kw)
            assert e.value.code == pkg.SARA_EINVAL


def test_kv_pool_exhaustion_and_exact_fit(pkg):
    """The paged KV cache: a pool smaller than one round's rollouts returns SARA_ENOMEM (and the
    handle stays usable); a pool of exactly the peak the step reported runs the step again with
    the same schedule and tokens -- the cache needs blocks for live positions only."""
    w = synth.WORKLOADS["tiny"]
    weights = synth.model_weights(w.model, w.weight_seed)
    si = synth.step_inputs(w)
    with pkg.Handle(handle_cfg(w, pkg), weights) as h:
        ref = h.collect_step(thresholds=si.thresholds, lengths=si.lengths, tokens=si.tokens, N=w.budget_N, k=w.k,
                             n0=w.n0, tau=w.tau, target_B=w.target_B, reward_seed=w.reward_seed,
                             sample_seed=w.sample_seed, want_tokens=True)
    # every tiny rollout (prompt 32 + at most 32 tokens) lives in one private block: the peak is
    # the largest round, the probe round of B x n0 rollouts
    assert ref.kv_blocks_peak == w.target_B * w.n0
    small = handle_cfg(w, pkg)
    small.kv_blocks = ref.kv_blocks_peak - 1
    with pkg.Handle(small, weights) as h:
        with pytest.raises(pkg.SaraError) as e:
            _step(h, w, si)
        assert e.value.code == pkg.SARA_ENOMEM
    exact = handle_cfg(w, pkg)
    exact.kv_blocks = ref.kv_blocks_peak
    with pkg.Handle(exact, weights) as h:
        out = h.collect_step(thresholds=si.thresholds, lengths=si.lengths, tokens=si.tokens, N=w.budget_N, k=w.k,
                             n0=w.n0, tau=w.tau, target_B=w.target_B, reward_seed=w.reward_seed,
                             sample_seed=w.sample_seed, want_tokens=True)
    _assert_oracle_schedule(out, w, si)
    assert out.kv_blocks_peak == ref.kv_blocks_peak
    for q in range(w.n_prompts):
        for j in range(int(out.n[q])):
            L = int(si.lengths[q, j])
            assert np.array_equal(out.tokens[q, j, :L], ref.tokens[q, j, :L])
