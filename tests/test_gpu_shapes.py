"""Decode-step parity beyond the workload shapes: more than 64 live rows (the GEMMs' M = 128
path), several attention units per CTA with split merges, and other head geometries (head
dim 64 with a 4-query group; a 1-query group at head dim 128).  Teacher-forced logits through
the C ABI against the float64 oracle, within the stated tolerance; sampled tokens equal the
oracle's Gumbel-max draw wherever the margin is clear."""
import numpy as np
import pytest

import synth
from gpu_util import LOGIT_MAX_ABS, LOGIT_REL_L2, logit_errors
from oracle import decode as o2

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def pkg():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_26253_gb300 as p
    p.load()
    return p


def _teacher_case(pkg, shape, n, Lp, T, seed):
    weights = synth.model_weights(shape, seed)
    rng = np.random.default_rng(seed + 11)
    prompts = rng.integers(0, shape.vocab, size=(n, Lp)).astype(np.int32)
    forced = rng.integers(0, shape.vocab, size=(n, T)).astype(np.int32)
    uids = (np.arange(n, dtype=np.int64) * 64 + 3)
    cfg = pkg.model_cfg(shape, max_prompts=n, max_active=n, max_seqs=n, max_prompt_len=Lp, max_gen_len=T + 1,
                        max_k=2)
    with pkg.Handle(cfg, weights) as h:
        logits, sampled = h.teacher_force(prompts, forced, uids, sample_seed=9)
    want = o2.teacher_forced_logits_batch(o2.Weights(shape, weights), prompts, forced)
    err, rel = logit_errors(logits, want)
    assert err < LOGIT_MAX_ABS and rel < LOGIT_REL_L2, (err, rel)
    for i in range(n):
        for t in range(T):
            tok, margin = o2.sample_token(logits[i, t], 9, int(uids[i]), t)
            if margin > 1e-4:
                assert sampled[i, t] == tok, (i, t)


def test_many_rows_and_long_prompts_tiny(pkg):
    # 80 rows (> 64: M = 128 GEMMs); 300-token prompts: 3 attention splits per row and kv
    # head -> 480 units over the CTAs (several per CTA, both warp groups, split merges)
    _teacher_case(pkg, synth.TINY, n=80, Lp=300, T=3, seed=0)


SMALL_HD64_G4 = synth.ModelShape("hd64-g4", layers=2, d_model=256, n_heads=4, n_kv_heads=1, head_dim=64, ffn=512,
                                 vocab=1024)
SMALL_HD128_G1 = synth.ModelShape("hd128-g1", layers=2, d_model=256, n_heads=2, n_kv_heads=2, head_dim=128,
                                  ffn=384, vocab=640)


@pytest.mark.parametrize("shape", [SMALL_HD64_G4, SMALL_HD128_G1], ids=lambda s: s.name)
def test_head_geometries(pkg, shape):
    _teacher_case(pkg, shape, n=24, Lp=140, T=3, seed=4)
