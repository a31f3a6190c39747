"""Shared helpers of the GPU parity tests (inputs from synth, expectations from oracle/)."""
import numpy as np

LOGIT_MAX_ABS = 3e-2   # per-step logits under teacher forcing (the stated parity tolerance)
LOGIT_REL_L2 = 1e-2


def handle_cfg(w, pkg, max_seqs=None, max_prompts=None):
    return pkg.model_cfg(w.model, max_prompts=max_prompts or w.n_prompts, max_active=w.target_B,
                         max_seqs=max_seqs or w.target_B * w.n0, max_prompt_len=w.prompt_len,
                         max_gen_len=w.lengths.max_len, max_k=w.k)


def logit_errors(got, want):
    err = float(np.abs(got - want).max())
    rel = float(np.linalg.norm(got - want) / np.linalg.norm(want))
    return err, rel
