"""Pins of the decode oracle O2 (oracle/decode.py) against independent routes.

Each model piece is checked against a library routine or a different formulation
(torch's scaled_dot_product_attention and rms_norm in float64, complex-exponential
rotary embedding), the whole forward against a torch float64 composition of those
routines, plus invariants (causality, zero-weight reductions) and the sampler
against the Gumbel distribution and softmax frequencies.
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import synth
from oracle import decode as o2


def test_attention_matches_torch_sdpa_gqa():
    rng = np.random.default_rng(0)
    for T, H, KVH, hd in [(1, 4, 2, 8), (7, 6, 1, 16), (33, 12, 2, 32), (20, 8, 8, 4)]:
        q = rng.standard_normal((T, H, hd))
        k = rng.standard_normal((T, KVH, hd))
        v = rng.standard_normal((T, KVH, hd))
        ours = o2.causal_gqa_attention(q, k, v)
        tq, tk, tv = (torch.from_numpy(a).permute(1, 0, 2)[None] for a in (q, k, v))
        ref = F.scaled_dot_product_attention(tq, tk, tv, is_causal=True, enable_gqa=True)
        np.testing.assert_allclose(ours, ref[0].permute(1, 0, 2).numpy(), rtol=1e-12, atol=1e-12)


def test_rmsnorm_matches_torch():
    rng = np.random.default_rng(1)
    x = rng.standard_normal((5, 64)) * 3
    g = rng.standard_normal(64)
    ref = F.rms_norm(torch.from_numpy(x), (64,), torch.from_numpy(g), eps=1e-6).numpy()
    np.testing.assert_allclose(o2.rmsnorm(x, g, 1e-6), ref, rtol=1e-12, atol=1e-12)


def test_rope_matches_complex_rotation():
    # pair (x_i, x_{i+hd/2}) as the complex number x_i + i x_{i+hd/2}, times e^{i pos theta^(-2i/hd)}
    rng = np.random.default_rng(2)
    T, Hh, hd, theta = 9, 3, 16, 1.0e6
    x = rng.standard_normal((T, Hh, hd))
    pos = np.arange(T) * 37 + 5
    half = hd // 2
    z = x[..., :half] + 1j * x[..., half:]
    w = np.exp(1j * np.outer(pos, theta ** (-np.arange(0, hd, 2) / hd)))[:, None, :]
    ref = z * w
    out = o2.rope(x, pos, theta)
    np.testing.assert_allclose(out[..., :half], ref.real, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(out[..., half:], ref.imag, rtol=1e-12, atol=1e-12)
    # relative-position property: <rope(q, p), rope(k, p')> depends only on p - p'
    q, k = rng.standard_normal((1, 1, hd)), rng.standard_normal((1, 1, hd))
    d1 = np.sum(o2.rope(q, np.array([10]), theta) * o2.rope(k, np.array([3]), theta))
    d2 = np.sum(o2.rope(q, np.array([1010]), theta) * o2.rope(k, np.array([1003]), theta))
    assert abs(d1 - d2) < 1e-9


def _torch_forward(W: o2.Weights, tokens: np.ndarray) -> np.ndarray:
    """Independent float64 composition from torch library routines (SDPA, rms_norm, silu,
    complex rotary embedding)."""
    m = W.m
    f = lambda b: torch.from_numpy(synth.bf16_bits_to_f32(b).astype(np.float64))
    T = tokens.size
    x = f(W.g["embed"])[torch.from_numpy(tokens.astype(np.int64))]
    pos = torch.arange(T, dtype=torch.float64)
    inv = m.rope_theta ** (-torch.arange(0, m.head_dim, 2, dtype=torch.float64) / m.head_dim)
    rot = torch.polar(torch.ones(T, m.head_dim // 2, dtype=torch.float64), torch.outer(pos, inv))

    def rope(t):  # t [heads, T, hd]
        half = m.head_dim // 2
        z = torch.complex(t[..., :half], t[..., half:]) * rot
        return torch.cat([z.real, z.imag], -1)

    for l in range(m.layers):
        L = W.layer(l)
        h = F.rms_norm(x, (m.d_model,), f(L["attn_norm"]), eps=m.rms_eps)
        q = (h @ f(L["wq"]).T).view(T, m.n_heads, m.head_dim).transpose(0, 1)
        k = (h @ f(L["wk"]).T).view(T, m.n_kv_heads, m.head_dim).transpose(0, 1)
        v = (h @ f(L["wv"]).T).view(T, m.n_kv_heads, m.head_dim).transpose(0, 1)
        o = F.scaled_dot_product_attention(rope(q)[None], rope(k)[None], v[None], is_causal=True,
                                           enable_gqa=True)[0]
        x = x + o.transpose(0, 1).reshape(T, -1) @ f(L["wo"]).T
        h = F.rms_norm(x, (m.d_model,), f(L["mlp_norm"]), eps=m.rms_eps)
        x = x + (F.silu(h @ f(L["wgate"]).T) * (h @ f(L["wup"]).T)) @ f(L["wdown"]).T
    x = F.rms_norm(x, (m.d_model,), f(W.g["final_norm"]), eps=m.rms_eps)
    return (x @ f(W.g["lm_head"]).T).numpy()


@pytest.fixture(scope="module")
def tiny_weights():
    return o2.Weights(synth.TINY, synth.model_weights(synth.TINY, 0))


def test_forward_matches_torch_composition(tiny_weights):
    toks = np.random.default_rng(3).integers(0, synth.TINY.vocab, 40)
    ours = o2.forward_logits(tiny_weights, toks)[0]
    np.testing.assert_allclose(ours, _torch_forward(tiny_weights, toks), rtol=1e-10, atol=1e-10)


def test_forward_is_causal(tiny_weights):
    rng = np.random.default_rng(4)
    a = rng.integers(0, synth.TINY.vocab, 30)
    b = a.copy()
    b[20:] = rng.integers(0, synth.TINY.vocab, 10)
    la = o2.forward_logits(tiny_weights, a)[0]
    lb = o2.forward_logits(tiny_weights, b)[0]
    np.testing.assert_array_equal(la[:20], lb[:20])
    assert np.abs(la[20:] - lb[20:]).max() > 1e-3


def test_zero_projections_reduce_to_embedding_readout():
    # W_o = W_down = 0: each layer is the identity on the residual stream, so
    # logits = RMSNorm(E[tok]) W_lm^T for every position.
    m = synth.TINY
    w = synth.model_weights(m, 0)
    for L in w["layers"]:
        L["wo"] = np.zeros_like(L["wo"])
        L["wdown"] = np.zeros_like(L["wdown"])
    W = o2.Weights(m, w)
    toks = np.array([5, 77, 300, 511])
    e = synth.bf16_bits_to_f32(w["embed"][toks]).astype(np.float64)
    want = (e / np.sqrt((e * e).mean(1, keepdims=True) + m.rms_eps)) @ \
        synth.bf16_bits_to_f32(w["lm_head"]).astype(np.float64).T
    np.testing.assert_allclose(o2.forward_logits(W, toks)[0], want, rtol=1e-12, atol=1e-12)


def test_single_token_attention_returns_value_projection():
    rng = np.random.default_rng(5)
    q = rng.standard_normal((1, 4, 8))
    k = rng.standard_normal((1, 2, 8))
    v = rng.standard_normal((1, 2, 8))
    out = o2.causal_gqa_attention(q, k, v)
    np.testing.assert_allclose(out[0, :2], np.repeat(v[0, :1], 2, 0))
    np.testing.assert_allclose(out[0, 2:], np.repeat(v[0, 1:], 2, 0))


def test_teacher_forcing_reproduces_sampled_rollout(tiny_weights):
    prompt = np.random.default_rng(6).integers(0, synth.TINY.vocab, 12)
    toks, margins, logits = o2.generate(tiny_weights, prompt, 6, sample_seed=5, uid=o2.uid_of(3, 1))
    tf = o2.teacher_forced_logits(tiny_weights, prompt, toks)
    np.testing.assert_allclose(tf, logits, rtol=1e-12, atol=1e-12)
    tfb = o2.teacher_forced_logits_batch(tiny_weights, prompt[None], toks[None])
    np.testing.assert_allclose(tfb[0], logits, rtol=1e-12, atol=1e-12)
    assert np.all(margins >= 0)


def test_gumbel_noise_distribution():
    g = np.concatenate([o2.gumbel_noise(9, uid, t, 4096) for uid in range(5) for t in range(5)])
    assert g.dtype == np.float32
    # Gumbel(0,1): mean = Euler-Mascheroni constant, variance = pi^2 / 6
    assert abs(g.mean() - 0.5772156649) < 4 * math.sqrt(math.pi ** 2 / 6 / g.size)
    assert abs(g.var() - math.pi ** 2 / 6) < 0.05
    # distinct keys give distinct streams
    assert not np.array_equal(o2.gumbel_noise(9, 0, 0, 64), o2.gumbel_noise(9, 0, 1, 64))
    assert not np.array_equal(o2.gumbel_noise(9, 0, 0, 64), o2.gumbel_noise(9, 1, 0, 64))


def test_gumbel_max_samples_softmax():
    logits = np.array([1.0, 0.0, -1.0, 2.0, 0.5, -3.0])
    p = np.exp(logits - logits.max())
    p /= p.sum()
    n = 30000
    counts = np.zeros(logits.size)
    for i in range(n):
        counts[o2.sample_token(logits, 11, i // 64, i % 64)[0]] += 1
    chi2 = float((((counts - n * p) ** 2) / (n * p)).sum())
    assert chi2 < 25.0  # 5 degrees of freedom; P(chi2 > 25) ~ 1e-4
    # a dominant logit always wins
    big = np.zeros(100)
    big[42] = 60.0
    assert all(o2.sample_token(big, 1, u, 0)[0] == 42 for u in range(50))


def test_attention_after_a_cached_prefix_equals_the_full_causal_attention():
    rng = np.random.default_rng(7)
    Tall, past, H, KVH, hd = 23, 15, 6, 2, 8
    q = rng.standard_normal((Tall, H, hd))
    k = rng.standard_normal((Tall, KVH, hd))
    v = rng.standard_normal((Tall, KVH, hd))
    full = o2.causal_gqa_attention(q, k, v)
    tail = o2.gqa_attention_after(q[past:], k, v, past)
    assert np.allclose(tail, full[past:], rtol=0, atol=1e-13)


def test_shared_prefix_teacher_forcing_equals_full_recompute(tiny_weights):
    W = tiny_weights
    rng = np.random.default_rng(8)
    V = W.m.vocab
    prefix = rng.integers(0, V, 21)
    suffixes = rng.integers(0, V, (3, 4))
    forced = rng.integers(0, V, (3, 5))
    got = o2.teacher_forced_logits_shared_prefix(W, prefix, suffixes, forced)
    prompts = np.concatenate([np.tile(prefix, (3, 1)), suffixes], axis=1)
    want = o2.teacher_forced_logits_batch(W, prompts, forced)
    assert got.shape == want.shape == (3, 5, V)
    assert np.abs(got - want).max() < 1e-11 * np.abs(want).max()
