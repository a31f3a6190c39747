"""End-to-end parity of the decode path through the C ABI.

Tiny config: the whole step (schedule bit-exact against O1, every decode step run, every
generated token equal to the oracle's Gumbel-max draw up to the first near-tie) and
teacher-forced logits.  1.5B / 3B shapes: teacher-forced logits on a slice of decode steps
within the tolerance, the fused sampler against the oracle sampler on the same logits, and
the whole step's schedule bit-exact."""
from dataclasses import replace

import numpy as np
import pytest

import synth
from gpu_util import LOGIT_MAX_ABS, LOGIT_REL_L2, handle_cfg, logit_errors
from oracle import controller as oc
from oracle import decode as o2

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def pkg():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_26253_gb300 as p
    p.load()
    return p


@pytest.fixture(scope="module")
def tiny(pkg):
    w = synth.WORKLOADS["tiny"]
    weights = synth.model_weights(w.model, w.weight_seed)
    h = pkg.Handle(handle_cfg(w, pkg), weights)
    yield w, weights, h
    h.close()


def _run_step(h, w, si, **kw):
    return h.collect_step(thresholds=si.thresholds, lengths=si.lengths, tokens=si.tokens, N=w.budget_N, k=w.k,
                          n0=w.n0, tau=w.tau, target_B=w.target_B, reward_seed=w.reward_seed,
                          sample_seed=w.sample_seed, commit_min=w.commit_floor, prior=w.prior, **kw)


def _assert_schedule(out, ref):
    assert np.array_equal(out.status, ref.status)
    assert np.array_equal(out.n, ref.n) and np.array_equal(out.s, ref.s)
    assert np.array_equal(out.decided_round, ref.decided_round)
    for key, v in ref.counters.items():
        assert out.counters[key] == v, (key, out.counters[key], v)


def test_tiny_step_schedule_and_tokens(tiny):
    w, weights, h = tiny
    si = synth.step_inputs(w)
    out = _run_step(h, w, si, want_tokens=True)
    ref = oc.collect_workload(w, si)
    _assert_schedule(out, ref)
    W = o2.Weights(w.model, weights)
    compared = 0
    for q in np.nonzero(ref.n)[0]:
        for j in range(int(ref.n[q])):
            L = int(si.lengths[q, j])
            toks, margins, _ = o2.generate(W, si.tokens[q], L, w.sample_seed, o2.uid_of(int(q), j))
            got = out.tokens[q, j, :L]
            low = np.nonzero(margins < 1e-2)[0]
            cut = int(low[0]) if low.size else L  # from a near-tie on, the draws may legitimately differ
            assert np.array_equal(got[:cut], toks[:cut]), (q, j, got[:cut + 1], toks[:cut + 1])
            compared += cut
    # a near-tie (top-two Gumbel-max margin < 1e-2, ~60x the logit error of this shape) ends a
    # rollout's comparison; the top-two gap of 512 Gumbel scores is near Exp(1), so about 1 % of
    # the draws are near-ties and ~90 % of the tokens are compared on average
    print(f"compared {compared} of {out.counters['gen_tokens']} tokens")
    assert compared > 0.8 * out.counters["gen_tokens"]


def test_tiny_step_is_deterministic_and_reusable(tiny):
    w, _, h = tiny
    si = synth.step_inputs(w)
    a = _run_step(h, w, si, want_tokens=True)
    b = _run_step(h, w, si, want_tokens=True)
    assert a.counters == b.counters
    for q in range(w.n_prompts):
        for j in range(int(a.n[q])):
            L = int(si.lengths[q, j])
            assert np.array_equal(a.tokens[q, j, :L], b.tokens[q, j, :L])


def test_tiny_other_seeds_and_configs(tiny):
    w0, _, h = tiny
    for off in (100, 200, 300):
        for kw in ({}, {"commit_min": 4}, {"tau": 0.3, "n0": 1}, {"budget_N": 90}):
            w = replace(w0.with_seed_offset(off), **kw)
            si = synth.step_inputs(w)
            _assert_schedule(_run_step(h, w, si), oc.collect_workload(w, si))


@pytest.mark.parametrize("eager", [False, True])
def test_tiny_teacher_forced_logits(tiny, eager):
    w, weights, h = tiny
    si = synth.step_inputs(w)
    rng = np.random.default_rng(1)
    n, T = 16, 24
    prompts = si.tokens[:n]
    forced = rng.integers(0, w.model.vocab, size=(n, T)).astype(np.int32)
    uids = np.arange(n, dtype=np.int64) * 64 + 1
    h.set_limits(eager_softmax=eager)
    try:
        logits, sampled = h.teacher_force(prompts, forced, uids, w.sample_seed)
    finally:
        h.set_limits()
    want = o2.teacher_forced_logits_batch(o2.Weights(w.model, weights), prompts, forced)
    err, rel = logit_errors(logits, want)
    assert err < LOGIT_MAX_ABS and rel < LOGIT_REL_L2, (err, rel)
    for i in range(n):
        for t in range(T):
            tok, margin = o2.sample_token(logits[i, t], w.sample_seed, int(uids[i]), t)
            if margin > 1e-4:
                assert sampled[i, t] == tok


def test_invalid_token_rejected(tiny):
    w, _, h = tiny
    si = synth.step_inputs(w)
    bad = si.tokens.copy()
    bad[3, 5] = w.model.vocab  # out of range: rejected on the host before any launch
    import paper_2607_26253_gb300 as pkg
    with pytest.raises(pkg.SaraError):
        h.collect_step(thresholds=si.thresholds, lengths=si.lengths, tokens=bad, N=w.budget_N, k=w.k, n0=w.n0,
                       tau=w.tau, target_B=w.target_B, reward_seed=w.reward_seed)


@pytest.mark.parametrize("name", ["1.5b", "3b"])
def test_full_shape_teacher_forced_slice(pkg, name):
    w = synth.WORKLOADS[name]
    m = w.model
    weights = synth.model_weights(m, w.weight_seed)
    si = synth.step_inputs(w)
    n, T = 2, 3
    prompts = si.tokens[:n]
    forced = np.random.default_rng(2).integers(0, m.vocab, size=(n, T)).astype(np.int32)
    uids = np.array([5, 70], np.int64)
    with pkg.Handle(handle_cfg(w, pkg), weights) as h:
        logits, sampled = h.teacher_force(prompts, forced, uids, w.sample_seed)
    want = o2.teacher_forced_logits_batch(o2.Weights(m, weights), prompts, forced)
    err, rel = logit_errors(logits, want)
    assert err < LOGIT_MAX_ABS and rel < LOGIT_REL_L2, (err, rel)
    for i in range(n):
        for t in range(T):
            tok, margin = o2.sample_token(logits[i, t], w.sample_seed, int(uids[i]), t)
            if margin > 1e-4:
                assert sampled[i, t] == tok


def test_full_shape_step_schedule_1p5b(pkg):
    w = synth.WORKLOADS["1.5b"]
    weights = synth.model_weights(w.model, w.weight_seed)
    si = synth.step_inputs(w)
    with pkg.Handle(handle_cfg(w, pkg), weights) as h:
        out = _run_step(h, w, si, want_tokens=True)
    _assert_schedule(out, oc.collect_workload(w, si))
    for q in np.nonzero(out.n)[0][:8]:
        for j in range(int(out.n[q])):
            t = out.tokens[q, j, :si.lengths[q, j]]
            assert t.min() >= 0 and t.max() < w.model.vocab


# Long contexts at the full shapes: many rows over a 2,000-token shared prefix, so that the
# decode step runs the paths the benchmark runs -- 26 rows (one stacked hi/lo operand per
# k-step) and 80 rows (above 64: hi and lo as separate 128-row operands), attention units of
# several KV blocks and rows split over several units, merged by the last split to finish.  The
# oracle computes the prefix once (its keys and values are shared) and then every row's own
# positions; rows differ in their last 4 prompt tokens and in their forced tokens.
LONG_PREFIX, LONG_SUFFIX, LONG_T, LONG_ROWS = 2000, 4, 2, 80


@pytest.fixture(scope="module", params=["1.5b", "3b"])
def long_case(pkg, request):
    w = synth.WORKLOADS[request.param]
    m = w.model
    weights = synth.model_weights(m, w.weight_seed)
    rng = np.random.default_rng(20)
    prefix = rng.integers(0, m.vocab, LONG_PREFIX).astype(np.int32)
    suffixes = rng.integers(0, m.vocab, (LONG_ROWS, LONG_SUFFIX)).astype(np.int32)
    forced = rng.integers(0, m.vocab, (LONG_ROWS, LONG_T)).astype(np.int32)
    want = o2.teacher_forced_logits_shared_prefix(o2.Weights(m, weights), prefix, suffixes, forced)
    prompts = np.concatenate([np.tile(prefix, (LONG_ROWS, 1)), suffixes], axis=1)
    cfg = pkg.model_cfg(m, max_prompts=LONG_ROWS, max_active=LONG_ROWS, max_seqs=128,
                        max_prompt_len=prompts.shape[1], max_gen_len=8, max_k=w.k)
    h = pkg.Handle(cfg, weights)
    yield w, h, prompts, forced, want
    h.close()


# eager: the attention re-bases its running maximum at every KV block that raises it, so the
# rescale of the output accumulated in registers runs on most blocks (by default it runs
# only when a score exceeds the running maximum by more than 2^8, which these inputs never do)
@pytest.mark.parametrize("eager", [False, True])
@pytest.mark.parametrize("n", [26, LONG_ROWS])
def test_full_shape_long_context_teacher_forced(long_case, n, eager):
    w, h, prompts, forced, want = long_case
    uids = np.arange(n, dtype=np.int64) * 64 + 3
    h.set_limits(eager_softmax=eager)
    try:
        logits, sampled = h.teacher_force(prompts[:n], forced[:n], uids, w.sample_seed)
    finally:
        h.set_limits()
    err, rel = logit_errors(logits, want[:n])
    print(f"{w.model.name} rows {n} context {prompts.shape[1]} eager {eager}: max-abs {err:.2e} rel-L2 {rel:.2e}")
    assert err < LOGIT_MAX_ABS and rel < LOGIT_REL_L2, (err, rel)
    for i in range(n):
        for t in range(LONG_T):
            tok, margin = o2.sample_token(logits[i, t], w.sample_seed, int(uids[i]), t)
            if margin > 1e-4:
                assert sampled[i, t] == tok, (i, t)


# The asynchronous per-prompt schedule on the decode engine (no round barrier): every prompt is
# decided at the end of the decode step in which its batch finishes, and the rollouts it issues
# join the live rows at the next step.  The schedule must equal the asynchronous oracle's bit
# for bit (decision events in place of rounds) and every decoded token the float64 oracle's
# Gumbel-max draw up to the first near-tie.
def _assert_async_schedule(out, ref):
    assert np.array_equal(out.status, ref.status)
    assert np.array_equal(out.n, ref.n) and np.array_equal(out.s, ref.s)
    assert np.array_equal(out.decided_round.astype(np.int32), np.minimum(ref.decided_event, 32767))
    c = ref.counters
    for key, v in (("rollouts", c["rollouts"]), ("gen_tokens", c["gen_tokens"]), ("decode_steps", c["decode_steps"]),
                   ("rounds", c["events"]), ("committed", c["committed"]), ("abandoned", c["abandoned"]),
                   ("incomplete", c["incomplete"]), ("prompts_drawn", c["prompts_drawn"]),
                   ("prefill_tokens", c["prefill_tokens"])):
        assert out.counters[key] == v, (key, out.counters[key], v)


@pytest.mark.parametrize("schedule", [1, 2])
def test_tiny_async_schedule_and_tokens(tiny, schedule):
    from oracle import async_schedule as oa
    w, weights, h = tiny
    si = synth.step_inputs(w)
    out = _run_step(h, w, si, want_tokens=True, schedule=schedule)
    ref = oa.collect_workload(w, si, reserve=schedule == 2)
    _assert_async_schedule(out, ref)
    W = o2.Weights(w.model, weights)
    compared = 0
    for q in np.nonzero(ref.n)[0]:
        for j in range(int(ref.n[q])):
            L = int(si.lengths[q, j])
            toks, margins, _ = o2.generate(W, si.tokens[q], L, w.sample_seed, o2.uid_of(int(q), j))
            low = np.nonzero(margins < 1e-2)[0]
            cut = int(low[0]) if low.size else L
            assert np.array_equal(out.tokens[q, j, :cut], toks[:cut]), (q, j)
            compared += cut
    assert compared > 0.8 * out.counters["gen_tokens"]


def test_tiny_async_other_seeds_and_the_round_schedule_after(tiny):
    from oracle import async_schedule as oa
    w0, _, h = tiny
    for off in (100, 200):
        for kw in ({}, {"commit_min": 4}, {"budget_N": 90}):
            w = replace(w0.with_seed_offset(off), **kw)
            si = synth.step_inputs(w)
            for schedule in (1, 2):
                _assert_async_schedule(_run_step(h, w, si, schedule=schedule),
                                       oa.collect_workload(w, si, reserve=schedule == 2))
            _assert_schedule(_run_step(h, w, si), oc.collect_workload(w, si))  # the same handle, rounds again


def test_full_shape_async_step_1p5b(pkg):
    from oracle import async_schedule as oa
    w = synth.WORKLOADS["1.5b"]
    weights = synth.model_weights(w.model, w.weight_seed)
    si = synth.step_inputs(w)
    with pkg.Handle(handle_cfg(w, pkg), weights) as h:
        out = _run_step(h, w, si, want_tokens=True, schedule=2)
    _assert_async_schedule(out, oa.collect_workload(w, si, reserve=True))
    for q in np.nonzero(out.n)[0][:8]:
        for j in range(int(out.n[q])):
            t = out.tokens[q, j, :si.lengths[q, j]]
            assert t.min() >= 0 and t.max() < w.model.vocab
