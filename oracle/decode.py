"""O2 -- float64 CPU oracle of the policy's decode path and its sampler.

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).

The paper generates rollouts with R1-Distill-Qwen-1.5B / Qwen2.5-3B in bf16
(App. E) at temperature 1.0 over the full vocabulary, but defines no model
math; the readings used here (and by the CUDA path) are:
  * pre-norm decoder: x += Attn(RMSNorm(x)); x += MLP(RMSNorm(x));
    logits = RMSNorm(x) @ W_lm^T (untied lm_head, no biases);
  * RMSNorm(x) = x / sqrt(mean(x^2) + eps) * g, eps = 1e-6;
  * rotary embedding, rotate-half pairing (i, i + hd/2), angle pos * theta^(-2i/hd),
    theta = 1e6, positions 0-based from the first prompt token;
  * causal grouped-query attention, q head h reads kv head h // (H / KVH),
    scale 1/sqrt(hd);
  * SwiGLU MLP: (silu(x W_g^T) * (x W_u^T)) W_d^T, silu(z) = z / (1 + e^-z);
  * a rollout of length L is L forward positions whose inputs are the last
    prompt token followed by its own first L-1 sampled tokens;
  * sampling at T = 1.0 is Gumbel-max: token = argmax_v (logit_v + g_v) with
    g_v = -log(-log(u_v)) and u_v from SplitMix64 in counter mode, decided in
    float32 (the precision the kernel decides in).
Everything here is computed in float64 with no blocking or fusion.
"""
from __future__ import annotations

import numpy as np

import synth

GOLDEN = np.uint64(0x9E3779B97F4A7C15)


# ------------------------------------------------------------------ model pieces
def rmsnorm(x: np.ndarray, g: np.ndarray, eps: float) -> np.ndarray:
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * g


def rope(x: np.ndarray, pos: np.ndarray, theta: float) -> np.ndarray:
    """x [T, heads, hd]; rotate pairs (i, i + hd/2) by pos * theta^(-2i/hd)."""
    hd = x.shape[-1]
    half = hd // 2
    inv_freq = theta ** (-(2.0 * np.arange(half, dtype=np.float64)) / hd)
    ang = pos.astype(np.float64)[:, None] * inv_freq[None, :]
    cos = np.cos(ang)[:, None, :]
    sin = np.sin(ang)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * cos - x2 * sin, x2 * cos + x1 * sin], axis=-1)


def causal_gqa_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray) -> np.ndarray:
    """q [T, H, hd], k/v [T, KVH, hd] -> [T, H, hd]; softmax(q k^T / sqrt(hd)) v, causal."""
    return gqa_attention_after(q, k, v, 0)


def gqa_attention_after(q: np.ndarray, k: np.ndarray, v: np.ndarray, past: int) -> np.ndarray:
    """Causal attention of queries at positions past .. past + T - 1: q [T, H, hd] against the
    keys / values of positions 0 .. past + T - 1, k/v [past + T, KVH, hd] -> [T, H, hd];
    query i sees keys 0 .. past + i."""
    T, H, hd = q.shape
    kvh = k.shape[1]
    group = H // kvh
    out = np.empty_like(q)
    mask = np.triu(np.ones((T, k.shape[0]), dtype=bool), past + 1)
    for h in range(H):
        kh = h // group
        sc = (q[:, h, :] @ k[:, kh, :].T) / np.sqrt(hd)
        sc[mask] = -np.inf
        sc -= sc.max(axis=1, keepdims=True)
        p = np.exp(sc)
        p /= p.sum(axis=1, keepdims=True)
        out[:, h, :] = p @ v[:, kh, :]
    return out


def silu(z: np.ndarray) -> np.ndarray:
    return z / (1.0 + np.exp(-z))


def _f64(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns -> float64 (float64 arrays pass through unchanged)."""
    if bits.dtype == np.float64:
        return bits
    return synth.bf16_bits_to_f32(bits).astype(np.float64)


def decoder_layer(x: np.ndarray, W: dict, m: synth.ModelShape, pos: np.ndarray, past=None, keep=None) -> np.ndarray:
    """One pre-norm decoder layer on one sequence x [T, d] at positions pos.  past: the
    (k, v) of this layer for the positions before pos[0] (a cached prefix), or None; keep: a
    list that receives this call's (k, v) after RoPE."""
    T = x.shape[0]
    hd = m.head_dim
    h = rmsnorm(x, _f64(W["attn_norm"]), m.rms_eps)
    q = (h @ _f64(W["wq"]).T).reshape(T, m.n_heads, hd)
    k = (h @ _f64(W["wk"]).T).reshape(T, m.n_kv_heads, hd)
    v = (h @ _f64(W["wv"]).T).reshape(T, m.n_kv_heads, hd)
    q = rope(q, pos, m.rope_theta)
    k = rope(k, pos, m.rope_theta)
    if keep is not None:
        keep.append((k, v))
    if past is None:
        o = causal_gqa_attention(q, k, v)
    else:
        o = gqa_attention_after(q, np.concatenate([past[0], k]), np.concatenate([past[1], v]), past[0].shape[0])
    o = o.reshape(T, m.n_heads * hd)
    x = x + o @ _f64(W["wo"]).T
    h2 = rmsnorm(x, _f64(W["mlp_norm"]), m.rms_eps)
    a = silu(h2 @ _f64(W["wgate"]).T) * (h2 @ _f64(W["wup"]).T)
    return x + a @ _f64(W["wdown"]).T


class Weights:
    """Weights by layer: a full synth.model_weights dict, or generated lazily from the seed."""

    def __init__(self, m: synth.ModelShape, weights: dict | None = None, seed: int = 0):
        self.m, self.seed = m, seed
        self.w = weights
        self.g = weights if weights is not None else synth.global_weights(m, seed)

    def layer(self, l: int) -> dict:
        if self.w is not None:
            return self.w["layers"][l]
        return synth.layer_weights(self.m, l, self.seed)


def forward_logits(W: Weights, tokens: np.ndarray, logit_positions=None) -> np.ndarray:
    """Causal forward of each sequence in tokens [S, T] (or [T]); returns float64 logits
    [S, len(logit_positions), V] for the requested positions (default: all)."""
    m = W.m
    toks = np.atleast_2d(np.asarray(tokens, dtype=np.int64))
    S, T = toks.shape
    sel = np.arange(T) if logit_positions is None else np.asarray(logit_positions)
    pos = np.arange(T)
    embed = W.g["embed"]
    xs = [_f64(embed[toks[i]]) for i in range(S)]
    for l in range(m.layers):
        Wl = W.layer(l)
        xs = [decoder_layer(x, Wl, m, pos) for x in xs]
    gf = _f64(W.g["final_norm"])
    lm = _f64(W.g["lm_head"])
    return np.stack([rmsnorm(x[sel], gf, m.rms_eps) @ lm.T for x in xs])


# ------------------------------------------------------------------ sampler
def _mix64(z: np.ndarray) -> np.ndarray:
    z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
    z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
    return z ^ (z >> np.uint64(31))


def gumbel_noise(sample_seed: int, uid: int, t: int, V: int) -> np.ndarray:
    """float32 Gumbel(0,1) noise for vocabulary entries of token t of rollout uid.

    Row seed = SplitMix64(sample_seed) output number uid * 2^20 + t + 1; entry v uses output
    number v + 1 of SplitMix64(row seed); u = (top 24 bits + 0.5) / 2^24; g = -log(-log u)."""
    row = synth.splitmix64_at(sample_seed, uid * (1 << 20) + t + 1)
    with np.errstate(over="ignore"):
        z = np.uint64(row) + (np.arange(1, V + 1, dtype=np.uint64) * GOLDEN)
        h = _mix64(z)
    u = (((h >> np.uint64(40)).astype(np.float32) + np.float32(0.5)) * np.float32(2.0 ** -24))
    return -np.log(-np.log(u))


def sample_token(logits_row: np.ndarray, sample_seed: int, uid: int, t: int) -> tuple[int, float]:
    """Gumbel-max over float32(logits); returns (token, margin between the top two scores)."""
    z = logits_row.astype(np.float32) + gumbel_noise(sample_seed, uid, t, logits_row.shape[-1])
    top2 = np.partition(z, -2)[-2:]
    return int(np.argmax(z)), float(top2[1] - top2[0])


def generate(W: Weights, prompt: np.ndarray, L: int, sample_seed: int, uid: int):
    """Autoregressive rollout: L tokens sampled at T=1 (full recompute each position).

    Returns (tokens [L], margins [L], logits [L, V])."""
    prompt = np.asarray(prompt, dtype=np.int64)
    seq = list(prompt)
    toks, margins, logits = [], [], []
    for t in range(L):
        lg = forward_logits(W, np.array(seq), logit_positions=[len(seq) - 1])[0, 0]
        tok, mg = sample_token(lg, sample_seed, uid, t)
        toks.append(tok)
        margins.append(mg)
        logits.append(lg)
        seq.append(tok)
    return np.array(toks, np.int32), np.array(margins), np.stack(logits)


def teacher_forced_logits(W: Weights, prompt: np.ndarray, forced: np.ndarray) -> np.ndarray:
    """Logits of decode steps 0..T-1 of a rollout whose generated tokens are `forced` [T]:
    step t sees prompt + forced[:t] and predicts forced[t]. Returns float64 [T, V]."""
    prompt = np.asarray(prompt, dtype=np.int64)
    forced = np.asarray(forced, dtype=np.int64)
    T = forced.size
    seq = np.concatenate([prompt, forced[:-1]]) if T > 0 else prompt
    Lp = prompt.size
    return forward_logits(W, seq, logit_positions=np.arange(Lp - 1, Lp - 1 + T))[0]


def uid_of(q: int, j: int) -> int:
    """Identity of rollout j of prompt q in the sampler's key."""
    return q * 64 + j


def teacher_forced_logits_batch(W: Weights, prompts: np.ndarray, forced: np.ndarray) -> np.ndarray:
    """teacher_forced_logits for S sequences at once: prompts [S, Lp], forced [S, T] -> [S, T, V]."""
    prompts = np.atleast_2d(np.asarray(prompts, dtype=np.int64))
    forced = np.atleast_2d(np.asarray(forced, dtype=np.int64))
    Lp, T = prompts.shape[1], forced.shape[1]
    seqs = np.concatenate([prompts, forced[:, :-1]], axis=1)
    return forward_logits(W, seqs, logit_positions=np.arange(Lp - 1, Lp - 1 + T))


def teacher_forced_logits_shared_prefix(W: Weights, prefix: np.ndarray, suffixes: np.ndarray,
                                        forced: np.ndarray) -> np.ndarray:
    """teacher_forced_logits_batch for prompts that share a long prefix: prompt i is
    prefix + suffixes[i] ([S, Ls]); forced [S, T] -> float64 [S, T, V].  The same forward as
    forward_logits: the prefix's keys and values of every layer are computed once and each
    sequence's later positions attend to them as they would in the full causal forward."""
    m = W.m
    prefix = np.asarray(prefix, dtype=np.int64)
    suffixes = np.atleast_2d(np.asarray(suffixes, dtype=np.int64))
    forced = np.atleast_2d(np.asarray(forced, dtype=np.int64))
    S, Ls = suffixes.shape
    T = forced.shape[1]
    Lc = prefix.size
    embed = W.g["embed"]
    # prefix: every layer's (k, v) after RoPE
    cache = []
    x = _f64(embed[prefix])
    pos = np.arange(Lc)
    for l in range(m.layers):
        keep = []
        x = decoder_layer(x, W.layer(l), m, pos, keep=keep)
        cache.append(keep[0])
    # each sequence's own positions Lc .. Lc + Ls + T - 2
    seqs = np.concatenate([suffixes, forced[:, :-1]], axis=1)
    n = seqs.shape[1]
    pos = Lc + np.arange(n)
    xs = [_f64(embed[seqs[i]]) for i in range(S)]
    for l in range(m.layers):
        Wl = {key: _f64(val) for key, val in W.layer(l).items()}  # converted once for all sequences
        xs = [decoder_layer(x, Wl, m, pos, past=cache[l]) for x in xs]
    gf = _f64(W.g["final_norm"])
    lm = _f64(W.g["lm_head"])
    sel = np.arange(Ls - 1, Ls - 1 + T)
    return np.stack([rmsnorm(x[sel], gf, m.rms_eps) @ lm.T for x in xs])
