/*
 * sara.h -- C ABI of the GB300 (sm_103a) rollout-collection library.
 *
 * The library runs one step of SARA, Sequential Adaptive Rollout Allocation
 * (arxiv 2607.26253), entirely on one GPU: batched bf16 autoregressive decode of
 * a decoder-only policy, interleaved with an on-device controller that keeps a
 * Beta posterior per prompt (Sec. 3.2), evaluates the closed-form effectiveness
 * predictor p_eff (Prop. 1, Eq. peff), applies the threshold rule (Eq. decide),
 * and refills freed slots from the prompt stream until B effective groups are
 * committed or the rollout budget N is spent (Algorithm 1).  Rewards are
 * synthetic and seeded, independent of the generated tokens.
 *
 * Conventions
 *   - Every function returns SARA_OK (0) or a negative SARA_E* code; no C++
 *     exception crosses this boundary.  sara_last_error() gives a message.
 *   - bf16 values travel as their uint16_t bit patterns.
 *   - Pointers marked "host or device" follow the struct's `on_device` flag:
 *     0 = host memory (pageable or pinned), 1 = device memory of the handle's GPU.
 *   - The library copies what it needs; the caller keeps ownership of every
 *     buffer it passes.  The handle owns all device state it allocates.
 *   - Work is issued on the CUDA stream given at creation (NULL = legacy default
 *     stream); calls return after that stream has finished the call's work.
 *   - One handle is used by one host thread at a time.
 */
#ifndef SARA_H
#define SARA_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define SARA_API __attribute__((visibility("default")))
#else
#define SARA_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* Layout version of the structs below.  Version 2 added sara_thresholds.schedule and decay,
 * sara_prompts.prior_a / prior_b, sara_model_cfg.kv_blocks, sara_result.decode_kernel_ms,
 * kv_blocks_peak and prior_a_next / prior_b_next, and sara_limits; version 3
 * sara_limits.eager_softmax;
 * a caller built against another version
 * must not pass its structs to this library (compare with sara_abi_version()). */
#define SARA_ABI_VERSION 3

#define SARA_OK 0
#define SARA_EINVAL (-1)   /* an argument is out of range; nothing was launched */
#define SARA_ENOMEM (-2)   /* device or host allocation failed, or a capacity is exceeded */
#define SARA_ETIMEOUT (-3) /* a bounded device wait or the step's iteration bound ran out */
#define SARA_EDEVICE (-4)  /* a CUDA call failed or a kernel reported an inconsistency */

/* Per-prompt outcome codes (sara_result.status). */
#define SARA_UNDRAWN 0     /* never drawn from the stream */
#define SARA_COMMITTED 2   /* effective group committed (mixed, size >= commit floor) */
#define SARA_ABANDONED 3   /* saturated prefix with p_eff < tau_low, or k all-same rollouts */
#define SARA_INCOMPLETE 4  /* drawn but left undecided when the step ended */

typedef struct sara_handle sara_handle;

/* Policy shape (a pre-norm decoder: RMSNorm, rotary GQA attention, SwiGLU MLP, untied
 * lm_head) and the capacities the handle allocates for. */
typedef struct {
    int32_t layers;          /* decoder layers; 0 creates a controller-only handle */
    int32_t d_model;         /* multiple of 128 */
    int32_t n_heads;         /* query heads */
    int32_t n_kv_heads;      /* key/value heads; n_heads / n_kv_heads in {1, 2, 4, 6, 8} */
    int32_t head_dim;        /* 32, 64 or 128 */
    int32_t ffn;             /* SwiGLU width, multiple of 64 */
    int32_t vocab;           /* multiple of 128 */
    float rope_theta;        /* rotary base, e.g. 1e6 */
    float rms_eps;           /* RMSNorm epsilon, e.g. 1e-6 */
    int32_t max_prompts;     /* largest prompt pool P per step */
    int32_t max_active;      /* largest target B (working-set size) per step, <= 8192 */
    int32_t max_seqs;        /* largest number of rollouts in one round (>= B * n0), <= 128 */
    int32_t max_prompt_len;  /* largest prompt length Lp */
    int32_t max_gen_len;     /* largest generated length of one rollout
                                (max_prompt_len + max_gen_len <= 12288) */
    int32_t max_k;           /* largest group size k (<= 64) */
    int32_t kv_blocks;       /* rollouts' private KV blocks of 128 positions in the paged cache
                                (0: enough for max_seqs rollouts of max_gen_len); a step that
                                needs more returns SARA_ENOMEM.  The prompts' full blocks are
                                held apart (max_active x (max_prompt_len - 1) / 128 of them) and
                                shared by each prompt's rollouts. */
} sara_model_cfg;

/* Policy weights, bf16 bit patterns, row-major [out_features][in_features] like a linear
 * layer's weight.  Per-layer fields are arrays of `layers` pointers.  Host or device
 * (on_device); copied into the handle by sara_create. */
typedef struct {
    const uint16_t *embed;                 /* [vocab][d_model] */
    const uint16_t *final_norm;            /* [d_model] */
    const uint16_t *lm_head;               /* [vocab][d_model] */
    const uint16_t *const *attn_norm;      /* [layers] x [d_model] */
    const uint16_t *const *wq;             /* [layers] x [n_heads*head_dim][d_model] */
    const uint16_t *const *wk;             /* [layers] x [n_kv_heads*head_dim][d_model] */
    const uint16_t *const *wv;             /* [layers] x [n_kv_heads*head_dim][d_model] */
    const uint16_t *const *wo;             /* [layers] x [d_model][n_heads*head_dim] */
    const uint16_t *const *mlp_norm;       /* [layers] x [d_model] */
    const uint16_t *const *wgate;          /* [layers] x [ffn][d_model] */
    const uint16_t *const *wup;            /* [layers] x [ffn][d_model] */
    const uint16_t *const *wdown;          /* [layers] x [d_model][ffn] */
    int32_t on_device;
} sara_weights;

/* The prompt pool D of Algorithm 1 in stream order (index = stream position). */
typedef struct {
    int32_t n_prompts;             /* P */
    int32_t prompt_len;            /* Lp (>= 2 with a model; any >= 1 controller-only) */
    const int32_t *tokens;         /* [P][Lp] token ids (unused controller-only; may be NULL) */
    const uint64_t *p_threshold;   /* [P] latent success rate as floor(p * 2^32); 2^32 = always */
    const int32_t *lengths;        /* [P][k] generated tokens of rollout j of prompt q, >= 1 */
    int32_t on_device;
    const double *prior_a;         /* [P] warm-start Beta prior of each prompt (App. D: its
                                      posterior carried from earlier steps), or NULL: every
                                      prompt starts from the integer prior of sara_thresholds */
    const double *prior_b;         /* [P], given together with prior_a; positive and finite.
                                      Decisions then compare p_eff in fp64 (log-Gamma), which
                                      agrees with exact arithmetic away from ties. */
} sara_prompts;

/* Decision-rule parameters (Eq. decide, App. D). */
typedef struct {
    int64_t tau_num, tau_den;  /* tau_low = tau_num / tau_den exactly, 0 <= tau_low <= 1,
                                  0 < tau_den < 2^31 (0.45 -> 9/20) */
    int32_t commit_min;        /* commit floor, 2..k; 0 means k (the paper's default) */
    int32_t alpha0, beta0;     /* integer Beta prior, each 1..8 (default 1, 1) */
    int32_t target_B;          /* effective groups wanted, 1..max_active */
    uint64_t sample_seed;      /* seed of the temperature-1 Gumbel-max sampler */
    int32_t schedule;          /* 0: synchronised rounds (Algorithm 1, the default);
                                  1: asynchronous per-prompt: a prompt is decided when its own
                                     rollouts finish and refill happens at the next decode step;
                                  2: as 1, drawing a fresh prompt only if the budget covers it
                                     and every prompt in flight running to k rollouts.
                                  On controller-only handles (layers == 0) decode time comes
                                  from the length table (decode_steps); on model handles the
                                  decode engine decides and refills at every decode-step
                                  boundary.  For 1 and 2, rounds counts the step boundaries
                                  with decisions and decided_round holds the index of the
                                  deciding one (capped at 32767).  Warm-start priors
                                  (sara_prompts.prior_a / prior_b) apply to every schedule. */
    double decay;              /* warm-start decay lambda in [0, 1] of the carried priors that
                                  sara_result.prior_a_next / prior_b_next receive */
} sara_thresholds;

/* Results of one step.  Array pointers may be NULL (not written); they are host or device
 * memory per `on_device`.  Counters are always written. */
typedef struct {
    uint8_t *status;           /* [P] SARA_* outcome */
    uint8_t *n;                /* [P] rollouts spent on the prompt */
    uint8_t *s;                /* [P] successes among them */
    int16_t *decided_round;    /* [P] round of the commit / abandon decision, else -1 */
    int32_t *tokens;           /* [P][k][max_gen_len] generated tokens of rollout (q, j),
                                  valid for j < n[q] and positions < lengths[q][j] */
    int32_t on_device;
    /* counters */
    int64_t rollouts;          /* rollouts generated (<= N) */
    int64_t gen_tokens;        /* sum of generated lengths */
    int64_t prefill_tokens;    /* prompt tokens prefilled ((Lp - 1) per drawn prompt) */
    int64_t decode_steps;      /* batched decode forward passes */
    int64_t rounds;            /* synchronisation rounds */
    int64_t committed, abandoned, incomplete, prompts_drawn;
    double device_ms;          /* GPU time of the step's kernels, inputs already on the device:
                                  CUDA events on the handle's stream after the input copies and
                                  before the output copies */
    double decode_kernel_ms;   /* summed duration of the decode-step kernel's launches (device
                                  clock, earliest CTA start to latest CTA end of each launch) */
    int64_t kv_blocks_peak;    /* most private KV blocks in use at once during the step */
    double *prior_a_next;      /* [P] or NULL (host or device per on_device): the next step's
                                  warm-start prior, alpha0 + decay (a - alpha0 + s) with a the
                                  prior this step used and s the prompt's successes */
    double *prior_b_next;      /* [P] or NULL: beta0 + decay (b - beta0 + n - s) */
} sara_result;

/*
 * Create a handle on the current CUDA device: allocate the KV cache, activation buffers and
 * controller state for the capacities in *cfg, copy the weights, build the step's CUDA graph.
 * weights may be NULL only when cfg->layers == 0 (controller-only handle).
 * stream: a cudaStream_t (or NULL) all later work is issued on.
 * Errors: SARA_EINVAL (shape or capacity out of range), SARA_ENOMEM, SARA_EDEVICE.
 */
SARA_API int sara_create(const sara_model_cfg *cfg, const sara_weights *weights, void *stream,
                         sara_handle **out);

/*
 * One rollout-collection step (Algorithm 1): probe, then per round decide -> refill ->
 * advance, with batched decode of every issued rollout, until |C| >= target_B, the budget N
 * is spent, or nothing can be issued.  The controller and the decode loop run on the GPU
 * without host round-trips (one graph launch with a device-evaluated loop condition).
 *   N: rollout budget cap (>= 0).  k: group size (2..min(64, max_k)).  n0: probe size (1..k).
 *   reward_seed: seed of the synthetic verdicts, verdict(q, j) = (SplitMix64 output number
 *     q*64 + j + 1 of reward_seed) >> 32 < p_threshold[q].
 * The step is stateless between calls apart from the weights.
 * Errors: SARA_EINVAL, SARA_ENOMEM (pool or round larger than the capacities),
 * SARA_ETIMEOUT, SARA_EDEVICE.
 */
SARA_API int sara_collect_step(sara_handle *h, const sara_prompts *prompts, int64_t N, int32_t k,
                               int32_t n0, const sara_thresholds *thr, uint64_t reward_seed,
                               sara_result *out);

/*
 * Teacher-forcing hook (testing): n_seq rollouts, rollout i with prompt prompts[i] (length
 * prompt_len) and generated tokens forced[i][0..T).  Runs the same prefill and decode
 * kernels as sara_collect_step; decode step t feeds the last prompt token (t = 0) or
 * forced[i][t-1] and writes its fp32 logits to logits[i][t][vocab] (host or device per
 * on_device) and, if sampled != NULL, the token the fused sampler drew for (uid[i], t)
 * with sample_seed into sampled[i][t].
 * Requires n_seq <= min(max_seqs, max_active), 2 <= prompt_len <= max_prompt_len,
 * 1 <= T <= max_gen_len.
 */
SARA_API int sara_teacher_force(sara_handle *h, int32_t n_seq, int32_t prompt_len,
                                const int32_t *prompts, int32_t T, const int32_t *forced,
                                const int64_t *uid, uint64_t sample_seed, float *logits,
                                int32_t *sampled, int32_t on_device);

/*
 * Profiling hook (benchmarks): set `rows` live rollouts at context length `ctx` (synthetic
 * row state; the step's own state is overwritten) and launch, after two warm-up launches,
 * `iters` copies of the decode step, captured in a CUDA graph (no host launch cost) and
 * timed with CUDA events on the handle's stream.  *ms_per_launch = elapsed / iters.
 *   kernel: 0 = whole decode step (the persistent decode-step kernel, then sampling and
 *               bookkeeping; positions advance by one per launch),
 *           1 = the decode-step kernel alone (embedding, every layer, lm_head with the
 *               Gumbel-max partials; positions fixed).
 * Requires 1 <= rows <= max_seqs, ctx >= 2 and room for the positions the launches use.
 */
SARA_API int sara_profile(sara_handle *h, int32_t kernel, int32_t rows, int32_t ctx, int32_t iters,
                          double *ms_per_launch);

/*
 * Failure limits (testing and watchdogs).  Every device wait of the step is bounded; these
 * fields tighten the bounds for later calls on the handle, so that the error paths can be
 * exercised without faulting or hanging the GPU.  All zero (stall_phase = -1) restores the
 * defaults.
 *   wait_limit_ns:  a bounded wait of the decode-step kernel gives up after this long and the
 *                   call returns SARA_ETIMEOUT (0: 2 s).
 *   max_loop_iters: the step's device loop ends with SARA_ETIMEOUT once it has run this many
 *                   iterations (0: only the built-in round bounds).
 *   stall_phase:    -1, or a phase-counter index of the decode-step kernel (0 = embedding,
 *                   1 + 9 l + j = phase j of layer l) whose waits are made to wait for a value
 *                   no launch reaches: they time out after wait_limit_ns.
 *   eager_softmax:  the decode attention's online softmax takes each KV block's
 *                   probabilities against a running maximum.  0 (default): the maximum is
 *                   re-based only when a probability against it would exceed 2^8, so
 *                   probabilities stay <= 256 and most blocks skip the block maximum and the
 *                   output rescale.  1: re-based at every block that raises it
 *                   (probabilities <= 1).  The same softmax up to rounding; the switch exists
 *                   to test the rescale path.
 * The handle stays usable after a call that failed this way.  SARA_EINVAL if out of range.
 */
typedef struct {
    int64_t wait_limit_ns;
    int32_t max_loop_iters;
    int32_t stall_phase;
    int32_t eager_softmax;
    int32_t reserved;        /* must be 0 */
} sara_limits;
SARA_API int sara_set_limits(sara_handle *h, const sara_limits *limits);

/* SARA_ABI_VERSION of the built library. */
SARA_API int sara_abi_version(void);

/* Message for the last error on this handle (or of sara_create when h == NULL). */
SARA_API const char *sara_last_error(const sara_handle *h);

/* Free the handle and all its device memory.  NULL is allowed. */
SARA_API void sara_destroy(sara_handle *h);

/* ---------------------------------------------------------------------------------------
 * Kernel-level entry points (device pointers, the caller's stream), for unit parity tests
 * of the building blocks.  The GEMM and the attention launch the kernels the step's prefill
 * of fresh prompts runs; the sampler is a one-CTA-per-row form of the decode step's
 * Gumbel-max.  The decode step itself runs its projections, attention and logits inside one
 * persistent kernel, which is tested end to end through sara_teacher_force.
 * ------------------------------------------------------------------------------------- */

/*
 * Y[r][n] = sum_c X[r][c] * W[n][c] for r < R, n < Nout (the prefill projection GEMM:
 * tcgen05 MMA with the accumulator in tensor memory, TMA-fed, stream-K over the weight).
 * X: [R][K] bf16, W: [Nout][K] bf16, Y: [R][Nout] fp32, all device, 16-byte aligned.
 * Shapes: 1 <= R <= 128, Nout % 128 == 0, K % 64 == 0, K >= 64.
 * workspace: device scratch of at least sara_gemm_workspace_bytes(R, Nout, K) bytes, all zero
 * on first use (the kernel leaves it zero again): per-CTA fixed-point tile sums and per-tile
 * arrival counters of the stream-K split.  Calls sharing a workspace must not overlap.
 */
SARA_API size_t sara_gemm_workspace_bytes(int32_t R, int32_t Nout, int32_t K);
SARA_API int sara_gemm_bf16(const uint16_t *X, const uint16_t *W, float *Y, int32_t R,
                            int32_t Nout, int32_t K, void *workspace, size_t workspace_bytes,
                            void *stream);

/*
 * The same GEMM as sara_gemm_bf16 for callers that cannot allocate device memory -- for
 * example code running inside a host framework whose memory pool has already reserved the
 * GPU (a raw cudaMalloc there fails or fragments the pool), or a plugin whose interface only
 * hands over inputs and outputs.  The paper has no counterpart; this is a library service.
 * It allocates nothing: the stream-K scratch is a fixed array inside the library
 * (8 MiB of tile sums for at most 64 CTAs + 8 KiB of tile counters), which every GPU that
 * loads the library holds until the process exits.  The first call on a device looks up
 * the array's device address (cudaGetSymbolAddress); make that first call before any
 * stream capture.  Every call shares the array: each call clears what it needs before its
 * kernel, and calls whose work overlaps on the GPU (several streams or threads) race and
 * must be serialised by the caller.  Shapes as sara_gemm_bf16, plus Nout <= 262,144
 * (SARA_EINVAL beyond).  X, W, Y device pointers; work is issued on `stream`.
 */
SARA_API int sara_gemm_bf16_static(const uint16_t *X, const uint16_t *W, float *Y, int32_t R,
                                   int32_t Nout, int32_t K, void *stream);

/*
 * Attention of b query rows against their own KV ranges (the prefill's attention kernel),
 * one query each (softmax(q K^T / sqrt(hd)) V with grouped-query heads): q [b][n_heads][hd] fp16; kv cache of sequence i at kv + i*kv_stride
 * elements, laid out [2 (K,V)][n_kv_heads][cap][hd] fp16, valid for positions < ctx[i];
 * out [b][n_heads][hd] bf16 (the high part of the step's bf16 hi/lo output pair).  Split over the context in chunks of 128 positions with an
 * fp32 log-sum-exp combine.  hd in {32, 64, 128}; n_heads / n_kv_heads in {1, 2, 4, 6, 8};
 * max_ctx <= 96 * 128.
 * workspace: >= sara_attention_workspace_bytes(b, n_heads, hd, max_ctx), counter area zero.
 */
SARA_API size_t sara_attention_workspace_bytes(int32_t b, int32_t n_heads, int32_t head_dim,
                                               int32_t max_ctx);
SARA_API int sara_attention_decode(const uint16_t *q, const uint16_t *kv, int64_t kv_stride,
                                   const int32_t *ctx, uint16_t *out, int32_t b, int32_t n_heads,
                                   int32_t n_kv_heads, int32_t head_dim, int32_t cap,
                                   int32_t max_ctx, void *workspace, size_t workspace_bytes,
                                   void *stream);

/*
 * Temperature-1 sampling by Gumbel-max (the decode step's sampling rule, one CTA per row):
 * token[r] = argmax_v (logits[r][v] + g(r, v)) with
 * g = -log(-log u), u from SplitMix64 keyed by (sample_seed, uid[r], t[r], v), decided in
 * fp32, ties to the lowest index.  logits [R][V] fp32, uid/t/token [R], all device.
 */
SARA_API int sara_sample(const float *logits, int32_t R, int32_t V, uint64_t sample_seed,
                         const int64_t *uid, const int32_t *t, int32_t *token, void *stream);

#ifdef __cplusplus
}
#endif
#endif /* SARA_H */
