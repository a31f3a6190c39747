// Device-resident state of one rollout-collection step: per-call constants, scalar
// progress variables, and the pointers every step kernel reads.  The whole step runs as
// one CUDA graph whose kernels take their sizes (live rows, items, prefill rows) from here.
#pragma once
#include <stdint.h>

namespace sara {

enum : uint8_t { ST_UNDRAWN = 0, ST_ACTIVE = 1, ST_COMMITTED = 2, ST_ABANDONED = 3, ST_INCOMPLETE = 4 };
enum : uint8_t { D_CONTINUE = 0, D_COMMIT = 1, D_ABANDON = 2 };

constexpr int kMaxK = 64;
constexpr int kTabDim = kMaxK + 1;  // tables indexed [n][s], 0 <= s <= n <= k

// Per-call constants (host -> device before the graph launch).
struct StepConst {
    int32_t P, Lp, k, n0, commit_min, a0, b0, B;
    int64_t N, tau_num, tau_den;
    uint64_t reward_seed, sample_seed;
    int32_t decode;       // 1: decode every issued rollout; 0: controller only
    int32_t teacher;      // 1: teacher forcing (one round, forced tokens)
    int32_t T_forced;     // teacher: generated tokens per rollout
    int32_t max_gen;      // stride of the generated-token output
    int32_t attn_chunk;   // decode attention: positions per KV block
    int32_t att_slots;    // decode attention: units one step runs at once, per kv head
    int32_t max_iters;    // bound on the step loop's iterations (0: none beyond the round bounds)
    int32_t stall_plus1;  // test hook: 1 + the decode-step phase counter whose waits never
                          // complete (0: none)
    int64_t wait_ns;      // limit of the decode step's bounded waits (0: the built-in 2 s)
    int32_t eager_softmax;  // 1: attention re-bases its running max at every block that raises it
    double tau_f;         // tau_num / tau_den (the warm-start predictor compares in fp64)
    int32_t warm;         // 1: per-prompt real priors q_pa / q_pb (warm-start) decide
    int32_t schedule;     // 0: synchronised rounds; 1 / 2: asynchronous per prompt (2: with the
                          // budget reserve), decided and refilled at every decode step
};

// Scalar progress of the step (device, reset by the init kernel).
struct StepVars {
    int32_t live;          // live decode rows
    int32_t att_items;     // decode attention work items
    int32_t pre_rows;      // prefill rows (fresh prompts x (Lp - 1))
    int32_t n_fresh;
    int32_t done;
    int32_t round;         // index of the round in flight (-1 before the probe)
    int32_t round_maxL;    // longest rollout of the round in flight
    int32_t round_steps;   // decode steps run in the round in flight
    int32_t n_act, n_iss;
    int32_t err;
    int32_t fin_count;     // arrival counter of the sample/finish kernel
    int32_t iters;         // loop iterations
    int32_t att_span;      // KV blocks per decode attention split of the next step
    int64_t used, C, cursor, drawn, gen_tokens, sched_steps, exec_steps, rounds_done;
    // decode-step kernel time: the launch in flight's earliest CTA start and latest CTA end
    // (globaltimer ns; kt0 = ~0 between launches), folded into kernel_ns by the bookkeeping
    unsigned long long kt0, kt1;
    int64_t kernel_ns;
    // paged KV cache: free private blocks on the stack, and the fewest ever free
    int32_t blk_top, blk_low;
    // new rollouts of this loop iteration (their slots in new_slots), for the KV set-up
    int32_t n_new;
    // asynchronous schedule: prompts whose batch finished in the last decode step (dec_list),
    // decision events so far, prompts with a batch in flight, the stop flag, free rollout slots
    // and prompt slots on their stacks, the budget held back for prompts in flight (reserve)
    int32_t n_dec, events, in_flight, stopped, slot_top, pslot_top;
    int64_t resv;
};

// KV blocks per decode attention split: the smallest span that leaves at most `slots` split
// units per kv head when `blocks` blocks (summed over the `rows` rows) are to be covered, and
// at least the rows' mean block count / kAttSplitsTarget, so that few long rows are not cut
// into many one-block splits (each split adds partial stores and a share of the merge).
constexpr int kAttSplitsTarget = 8;
__host__ __device__ inline int att_span_for(int64_t blocks, int slots, int64_t rows) {
    if (slots < 1) slots = 1;
    if (rows < 1) rows = 1;
    int64_t s = (blocks + slots - 1) / slots;
    const int64_t by_len = (blocks + rows * kAttSplitsTarget - 1) / (rows * kAttSplitsTarget);
    if (by_len > s) s = by_len;
    return s < 1 ? 1 : (int)s;
}

struct StepPtrs {
    StepConst *kc;
    StepVars *v;
    // prompt pool
    const int32_t *p_tok;      // [P][Lp]
    const uint64_t *p_thr;     // [P]
    const int32_t *p_len;      // [P][k]
    // per prompt
    uint8_t *q_status, *q_n, *q_s;
    int16_t *q_round;
    int32_t *q_pslot;
    // working lists
    int32_t *act, *act_tmp, *iss_q, *iss_c, *fresh_pslot;
    // exact decision / priority tables
    uint8_t *dec_tab, *rank_tab;
    // warm-start: per-prompt real Beta prior (used when StepConst::warm, else every prompt has
    // the integer prior of StepConst and the exact tables decide); p_eff keys of the continuing
    // prompts
    double *q_pa, *q_pb;
    double *q_key;
    // sequences (slots)
    int32_t *seq_q, *seq_j, *seq_len, *seq_gen, *seq_pslot;
    int64_t *seq_uid;
    // decode rows of the next step
    int32_t *row_slot, *row_pos, *row_tok, *row_item0;
    uint64_t *row_seed;
    int2 *att_items;
    int32_t *sampled;          // [max_seqs] token drawn for each row
    // prefill rows of the round
    int32_t *pre_slot, *pre_pos, *pre_tok, *pre_item0;
    int2 *pre_items;
    // outputs
    int32_t *gen_tok;          // [P][k][max_gen]
    // teacher forcing
    const int32_t *forced;     // [n][T]
    int32_t *sampled_out;      // [n][T]
    // sampling partial argmax per (row, vocabulary chunk)
    float *arg_val;
    int32_t *arg_idx;
    int32_t lm_tiles;
    int32_t max_seqs, max_active, pre_cap, att_cap;
    // paged KV cache of 128-position blocks.  Block ids [0, n_shared) hold the prompts' full
    // blocks (prompt slot ps owns ids ps * nsh_max ..), ids [n_shared, n_shared + n_priv) are
    // the rollouts' private blocks, handed out from the free stack blk_free[0, blk_top).
    int32_t *blk_tab;          // [max_seqs][nblk_max] block id of rollout slot s's block b
    int32_t *blk_free;         // [n_priv]
    int32_t nblk_max, nsh_max, n_shared, n_priv;
    int32_t *new_slots;        // [max_seqs] slots of the rollouts that start at the next step
    // asynchronous schedule
    int32_t *q_inflight;       // [P] rollouts of the prompt's batch still decoding
    int32_t *dec_list;         // [max_active] prompts to decide at this step boundary
    int32_t *slot_free;        // [max_seqs] free rollout slots
    int32_t *pslot_free;       // [max_active] free prompt slots
};

// Full prompt blocks (shared by a prompt's rollouts) when the prefill writes positions
// 0 .. Lp - 2; the block holding Lp - 1, the first decode position, is each rollout's own.
__host__ __device__ inline int shared_blocks(int Lp, int block) { return (Lp - 1) / block; }

}  // namespace sara
