"""ctypes binding of libsara.so (include/sara.h): argument marshalling only.

Every step of the rollout-collection path runs in the library's CUDA kernels.  Host
buffers are numpy arrays; device buffers are torch CUDA tensors (PyTorch supplies device
memory and streams only).  Loading fails loudly when the library has not been built.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from fractions import Fraction

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_build", "libsara.so")

SARA_OK, SARA_EINVAL, SARA_ENOMEM, SARA_ETIMEOUT, SARA_EDEVICE = 0, -1, -2, -3, -4
UNDRAWN, COMMITTED, ABANDONED, INCOMPLETE = 0, 2, 3, 4
EXPORTED = ("sara_create", "sara_collect_step", "sara_teacher_force", "sara_last_error", "sara_destroy",
            "sara_gemm_workspace_bytes", "sara_gemm_bf16", "sara_attention_workspace_bytes",
            "sara_attention_decode", "sara_sample", "sara_profile", "sara_gemm_bf16_static", "sara_set_limits",
            "sara_abi_version")
ABI_VERSION = 3

c_p = ctypes.c_void_p


class ModelCfg(ctypes.Structure):
    _fields_ = [("layers", ctypes.c_int32), ("d_model", ctypes.c_int32), ("n_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("ffn", ctypes.c_int32),
                ("vocab", ctypes.c_int32), ("rope_theta", ctypes.c_float), ("rms_eps", ctypes.c_float),
                ("max_prompts", ctypes.c_int32), ("max_active", ctypes.c_int32), ("max_seqs", ctypes.c_int32),
                ("max_prompt_len", ctypes.c_int32), ("max_gen_len", ctypes.c_int32), ("max_k", ctypes.c_int32),
                ("kv_blocks", ctypes.c_int32)]


class Weights(ctypes.Structure):
    _fields_ = [("embed", c_p), ("final_norm", c_p), ("lm_head", c_p), ("attn_norm", c_p), ("wq", c_p),
                ("wk", c_p), ("wv", c_p), ("wo", c_p), ("mlp_norm", c_p), ("wgate", c_p), ("wup", c_p),
                ("wdown", c_p), ("on_device", ctypes.c_int32)]


class Prompts(ctypes.Structure):
    _fields_ = [("n_prompts", ctypes.c_int32), ("prompt_len", ctypes.c_int32), ("tokens", c_p),
                ("p_threshold", c_p), ("lengths", c_p), ("on_device", ctypes.c_int32), ("prior_a", c_p),
                ("prior_b", c_p)]


class Thresholds(ctypes.Structure):
    _fields_ = [("tau_num", ctypes.c_int64), ("tau_den", ctypes.c_int64), ("commit_min", ctypes.c_int32),
                ("alpha0", ctypes.c_int32), ("beta0", ctypes.c_int32), ("target_B", ctypes.c_int32),
                ("sample_seed", ctypes.c_uint64), ("schedule", ctypes.c_int32), ("decay", ctypes.c_double)]


class Result(ctypes.Structure):
    _fields_ = [("status", c_p), ("n", c_p), ("s", c_p), ("decided_round", c_p), ("tokens", c_p),
                ("on_device", ctypes.c_int32), ("rollouts", ctypes.c_int64), ("gen_tokens", ctypes.c_int64),
                ("prefill_tokens", ctypes.c_int64), ("decode_steps", ctypes.c_int64), ("rounds", ctypes.c_int64),
                ("committed", ctypes.c_int64), ("abandoned", ctypes.c_int64), ("incomplete", ctypes.c_int64),
                ("prompts_drawn", ctypes.c_int64), ("device_ms", ctypes.c_double),
                ("decode_kernel_ms", ctypes.c_double), ("kv_blocks_peak", ctypes.c_int64),
                ("prior_a_next", c_p), ("prior_b_next", c_p)]


class Limits(ctypes.Structure):
    _fields_ = [("wait_limit_ns", ctypes.c_int64), ("max_loop_iters", ctypes.c_int32),
                ("stall_phase", ctypes.c_int32), ("eager_softmax", ctypes.c_int32), ("reserved", ctypes.c_int32)]


class SaraError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"sara error {code}: {msg}")
        self.code = code


_lib = None


def load(path: str = LIB_PATH):
    """Load libsara.so; raises if it has not been built (there is no fallback path)."""
    global _lib
    if _lib is not None and path == LIB_PATH:
        return _lib
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: build it with paper_2607_26253_gb300.build.build() "
                          "(or __graft_entry__.build()); there is no CPU fallback")
    lib = ctypes.CDLL(path)
    lib.sara_create.argtypes = [ctypes.POINTER(ModelCfg), ctypes.POINTER(Weights), c_p, ctypes.POINTER(c_p)]
    lib.sara_create.restype = ctypes.c_int
    lib.sara_collect_step.argtypes = [c_p, ctypes.POINTER(Prompts), ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                                      ctypes.POINTER(Thresholds), ctypes.c_uint64, ctypes.POINTER(Result)]
    lib.sara_collect_step.restype = ctypes.c_int
    lib.sara_teacher_force.argtypes = [c_p, ctypes.c_int32, ctypes.c_int32, c_p, ctypes.c_int32, c_p, c_p,
                                       ctypes.c_uint64, c_p, c_p, ctypes.c_int32]
    lib.sara_teacher_force.restype = ctypes.c_int
    lib.sara_last_error.argtypes = [c_p]
    lib.sara_last_error.restype = ctypes.c_char_p
    lib.sara_destroy.argtypes = [c_p]
    lib.sara_destroy.restype = None
    lib.sara_gemm_workspace_bytes.argtypes = [ctypes.c_int32] * 3
    lib.sara_gemm_workspace_bytes.restype = ctypes.c_size_t
    lib.sara_gemm_bf16.argtypes = [c_p, c_p, c_p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, c_p,
                                   ctypes.c_size_t, c_p]
    lib.sara_gemm_bf16.restype = ctypes.c_int
    lib.sara_attention_workspace_bytes.argtypes = [ctypes.c_int32] * 4
    lib.sara_attention_workspace_bytes.restype = ctypes.c_size_t
    lib.sara_attention_decode.argtypes = [c_p, c_p, ctypes.c_int64, c_p, c_p] + [ctypes.c_int32] * 6 + \
        [c_p, ctypes.c_size_t, c_p]
    lib.sara_attention_decode.restype = ctypes.c_int
    lib.sara_sample.argtypes = [c_p, ctypes.c_int32, ctypes.c_int32, ctypes.c_uint64, c_p, c_p, c_p, c_p]
    lib.sara_sample.restype = ctypes.c_int
    lib.sara_profile.argtypes = [c_p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                 ctypes.POINTER(ctypes.c_double)]
    lib.sara_profile.restype = ctypes.c_int
    lib.sara_gemm_bf16_static.argtypes = [c_p, c_p, c_p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, c_p]
    lib.sara_gemm_bf16_static.restype = ctypes.c_int
    lib.sara_set_limits.argtypes = [c_p, ctypes.POINTER(Limits)]
    lib.sara_set_limits.restype = ctypes.c_int
    lib.sara_abi_version.argtypes = []
    lib.sara_abi_version.restype = ctypes.c_int
    if lib.sara_abi_version() != ABI_VERSION:
        raise ImportError(f"{path} has ABI version {lib.sara_abi_version()}, this binding {ABI_VERSION}: rebuild it")
    if path == LIB_PATH:
        _lib = lib
    return lib


def _check(rc: int, handle=None):
    if rc != SARA_OK:
        msg = load().sara_last_error(handle)
        raise SaraError(rc, msg.decode() if msg else "")


def _ptr(a):
    """Address of a numpy array or torch tensor (None -> NULL)."""
    if a is None:
        return None
    if isinstance(a, np.ndarray):
        assert a.flags["C_CONTIGUOUS"], "arrays must be C-contiguous"
        return a.ctypes.data
    return a.data_ptr()


def tau_fraction(tau) -> Fraction:
    """tau_low as an exact rational: a Fraction as given, a float by its shortest decimal."""
    f = tau if isinstance(tau, Fraction) else Fraction(repr(float(tau)))
    if not (0 <= f <= 1) or f.denominator >= 2 ** 31:
        raise ValueError(f"tau_low must be a rational in [0, 1] with a 31-bit denominator: {tau}")
    return f


def model_cfg(shape, *, max_prompts: int, max_active: int, max_seqs: int, max_prompt_len: int,
              max_gen_len: int, max_k: int = 64, kv_blocks: int = 0) -> ModelCfg:
    """ModelCfg from a shape with fields layers, d_model, n_heads, n_kv_heads, head_dim, ffn, vocab,
    rope_theta, rms_eps (shape=None: controller-only handle)."""
    if shape is None:
        return ModelCfg(0, 0, 0, 0, 0, 0, 0, 0.0, 0.0, max_prompts, max_active, max_seqs, max_prompt_len,
                        max_gen_len, max_k, 0)
    return ModelCfg(shape.layers, shape.d_model, shape.n_heads, shape.n_kv_heads, shape.head_dim, shape.ffn,
                    shape.vocab, shape.rope_theta, shape.rms_eps, max_prompts, max_active, max_seqs,
                    max_prompt_len, max_gen_len, max_k, kv_blocks)


COUNTERS = ("rollouts", "gen_tokens", "prefill_tokens", "decode_steps", "rounds", "committed", "abandoned",
            "incomplete", "prompts_drawn")


@dataclass
class StepOutput:
    status: object
    n: object
    s: object
    decided_round: object
    tokens: object
    counters: dict
    device_ms: float          # the step's kernels, inputs already on the device
    decode_kernel_ms: float   # summed decode-step kernel launches (device clock)
    kv_blocks_peak: int       # most private KV blocks in use at once
    prior_next: tuple | None = None  # (a, b) warm-start priors of the next step, if requested


class Handle:
    """A sara_handle: model weights and every device buffer of the rollout-collection step."""

    def __init__(self, cfg: ModelCfg, weights: dict | None = None, stream=None):
        lib = load()
        keep = []
        wp = None
        if weights is not None:
            L = cfg.layers
            on_dev = not isinstance(weights["embed"], np.ndarray)

            def arr(name):
                ptrs = (c_p * L)(*[_ptr(weights["layers"][l][name]) for l in range(L)])
                keep.append(ptrs)
                return ctypes.cast(ptrs, c_p)

            w = Weights(_ptr(weights["embed"]), _ptr(weights["final_norm"]), _ptr(weights["lm_head"]),
                        arr("attn_norm"), arr("wq"), arr("wk"), arr("wv"), arr("wo"), arr("mlp_norm"),
                        arr("wgate"), arr("wup"), arr("wdown"), 1 if on_dev else 0)
            wp = ctypes.byref(w)
        self.cfg = cfg
        h = c_p()
        sp = None if stream is None else (stream.cuda_stream if hasattr(stream, "cuda_stream") else stream)
        _check(lib.sara_create(ctypes.byref(cfg), wp, sp, ctypes.byref(h)))
        self._h = h

    def close(self):
        if getattr(self, "_h", None):
            load().sara_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *a):
        self.close()

    def collect_step(self, *, thresholds, lengths, N: int, k: int, n0: int, tau, target_B: int,
                     reward_seed: int, tokens=None, prompt_len: int | None = None, commit_min: int = 0,
                     prior=(1, 1), sample_seed: int = 0, want_tokens: bool = False,
                     outputs_on_device: bool = False, schedule: int = 0, outputs: dict | None = None,
                     prior_a=None, prior_b=None, decay: float = 0.0, want_next_prior: bool = False) -> StepOutput:
        """One rollout-collection step (Algorithm 1).  Inputs are numpy arrays (host) or torch
        CUDA tensors (device); outputs are numpy arrays, or torch CUDA tensors when
        outputs_on_device.  `outputs` may hold preallocated arrays (keys status, n, s,
        decided_round and, with want_tokens, tokens [P, k, max_gen_len]) of the same kind.
        prior_a / prior_b: per-prompt warm-start priors (float64 [P], same kind as the inputs);
        want_next_prior: also return the next step's priors carried with `decay`."""
        P = int(thresholds.shape[0])
        on_dev = not isinstance(thresholds, np.ndarray)
        Lp = int(tokens.shape[1]) if tokens is not None else (prompt_len or 1)
        pr = Prompts(P, Lp, _ptr(tokens), _ptr(thresholds), _ptr(lengths), 1 if on_dev else 0, _ptr(prior_a),
                     _ptr(prior_b))
        t = tau_fraction(tau)
        th = Thresholds(t.numerator, t.denominator, commit_min, prior[0], prior[1], target_B, sample_seed, schedule,
                        float(decay))
        if outputs is not None:
            status, n, s, rnd = outputs["status"], outputs["n"], outputs["s"], outputs["decided_round"]
            toks = outputs["tokens"] if want_tokens else None
        elif outputs_on_device:
            import torch
            status = torch.zeros(P, dtype=torch.uint8, device="cuda")
            n = torch.zeros(P, dtype=torch.uint8, device="cuda")
            s = torch.zeros(P, dtype=torch.uint8, device="cuda")
            rnd = torch.zeros(P, dtype=torch.int16, device="cuda")
            toks = (torch.empty((P, k, self.cfg.max_gen_len), dtype=torch.int32, device="cuda")
                    if want_tokens else None)
        else:
            status = np.zeros(P, np.uint8)
            n = np.zeros(P, np.uint8)
            s = np.zeros(P, np.uint8)
            rnd = np.zeros(P, np.int16)
            toks = np.empty((P, k, self.cfg.max_gen_len), np.int32) if want_tokens else None
        pan = pbn = None
        if want_next_prior:
            if outputs_on_device:
                import torch
                pan = torch.empty(P, dtype=torch.float64, device="cuda")
                pbn = torch.empty(P, dtype=torch.float64, device="cuda")
            else:
                pan, pbn = np.empty(P, np.float64), np.empty(P, np.float64)
        res = Result(_ptr(status), _ptr(n), _ptr(s), _ptr(rnd), _ptr(toks), 1 if outputs_on_device else 0)
        res.prior_a_next, res.prior_b_next = _ptr(pan), _ptr(pbn)
        _check(load().sara_collect_step(self._h, ctypes.byref(pr), N, k, n0, ctypes.byref(th), reward_seed,
                                        ctypes.byref(res)), self._h)
        counters = {name: int(getattr(res, name)) for name in COUNTERS}
        return StepOutput(status, n, s, rnd, toks, counters, float(res.device_ms), float(res.decode_kernel_ms),
                          int(res.kv_blocks_peak), (pan, pbn) if want_next_prior else None)

    def set_limits(self, wait_limit_ns: int = 0, max_loop_iters: int = 0, stall_phase: int = -1,
                   eager_softmax: bool = False):
        """Failure limits of later calls (see sara_set_limits); no arguments restores the defaults."""
        lim = Limits(wait_limit_ns, max_loop_iters, stall_phase, int(eager_softmax), 0)
        _check(load().sara_set_limits(self._h, ctypes.byref(lim)), self._h)

    def profile(self, kernel: int, rows: int, ctx: int, iters: int = 20) -> float:
        """Milliseconds per launch of the decode step (kernel 0) or of the decode-step kernel
        alone (kernel 1); see sara_profile in include/sara.h."""
        ms = ctypes.c_double()
        _check(load().sara_profile(self._h, kernel, rows, ctx, iters, ctypes.byref(ms)), self._h)
        return ms.value

    def teacher_force(self, prompts: np.ndarray, forced: np.ndarray, uids: np.ndarray, sample_seed: int):
        """Logits [n, T, V] (fp32) and sampled tokens [n, T] of teacher-forced decode steps."""
        prompts = np.ascontiguousarray(prompts, np.int32)
        forced = np.ascontiguousarray(forced, np.int32)
        uids = np.ascontiguousarray(uids, np.int64)
        n, Lp = prompts.shape
        T = forced.shape[1]
        logits = np.empty((n, T, self.cfg.vocab), np.float32)
        sampled = np.empty((n, T), np.int32)
        _check(load().sara_teacher_force(self._h, n, Lp, _ptr(prompts), T, _ptr(forced), _ptr(uids), sample_seed,
                                         _ptr(logits), _ptr(sampled), 0), self._h)
        return logits, sampled


def gemm_bf16(X, W, workspace=None):
    """Y = X @ W^T (bf16 in, fp32 out) with the tcgen05 kernel; X [R, K], W [N, K] torch bf16 CUDA."""
    import torch
    R, K = X.shape
    N = W.shape[0]
    Y = torch.empty((R, N), dtype=torch.float32, device=X.device)
    if workspace is None:
        nbytes = load().sara_gemm_workspace_bytes(R, N, K)
        workspace = torch.zeros(nbytes, dtype=torch.uint8, device=X.device)
    _check(load().sara_gemm_bf16(X.data_ptr(), W.data_ptr(), Y.data_ptr(), R, N, K, workspace.data_ptr(),
                                 workspace.numel(), torch.cuda.current_stream().cuda_stream))
    return Y


def gemm_bf16_static(X, W, out=None):
    """Y = X @ W^T like gemm_bf16, through the entry point that allocates nothing (its scratch
    is a fixed array inside the library).  X [R, K], W [N, K] torch bf16 CUDA; `out` [R, N]
    fp32 CUDA may be passed so the call itself allocates nothing."""
    import torch
    R, K = X.shape
    N = W.shape[0]
    Y = out if out is not None else torch.empty((R, N), dtype=torch.float32, device=X.device)
    _check(load().sara_gemm_bf16_static(X.data_ptr(), W.data_ptr(), Y.data_ptr(), R, N, K,
                                        torch.cuda.current_stream().cuda_stream))
    return Y


def attention_decode(q, kv, ctx, n_kv_heads: int, cap: int, max_ctx: int | None = None):
    """Decode attention: q [b, H, hd] fp16, kv [b, 2, KVH, cap, hd] fp16, ctx [b] int32 (CUDA);
    returns bf16 [b, H, hd]."""
    import torch
    b, H, hd = q.shape
    max_ctx = int(ctx.max().item()) if max_ctx is None else max_ctx
    out = torch.empty(q.shape, dtype=torch.bfloat16, device=q.device)
    nbytes = load().sara_attention_workspace_bytes(b, H, hd, max_ctx)
    ws = torch.zeros(nbytes, dtype=torch.uint8, device=q.device)
    _check(load().sara_attention_decode(q.data_ptr(), kv.data_ptr(), kv.stride(0), ctx.data_ptr(), out.data_ptr(),
                                        b, H, n_kv_heads, hd, cap, max_ctx, ws.data_ptr(), ws.numel(),
                                        torch.cuda.current_stream().cuda_stream))
    return out


def sample(logits, uid, t, sample_seed: int):
    """Gumbel-max token per row of fp32 logits [R, V] (CUDA) keyed by (uid[r], t[r])."""
    import torch
    R, V = logits.shape
    tok = torch.empty(R, dtype=torch.int32, device=logits.device)
    _check(load().sara_sample(logits.data_ptr(), R, V, sample_seed, uid.data_ptr(), t.data_ptr(), tok.data_ptr(),
                              torch.cuda.current_stream().cuda_stream))
    return tok
