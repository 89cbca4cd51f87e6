/*
 * cai.h: C ABI of the GB300 (sm_103a) decoding head and commit controller
 * of CAI-dLLM, "Convergence Aware Inference for diffusion LLMs"
 * (arXiv 2608.22646).
 *
 * One denoising step, for the masked positions of the current output block of
 * every sequence in the batch:
 *   1. logits z = W h for each masked row (Box 1: p_theta(x_i | x^(t)) over the
 *      vocabulary), on tcgen05 tensor cores, never written to memory;
 *   2. the full-vocabulary softmax reduced to the confidence
 *      c_i = max_v p(v) and the greedy token argmax_v p(v) (Box 1, temperature 0
 *      per Section 5 "Setup");
 *   3. the commit rule of Algorithm 1: first-step confidence s_i (Box 2),
 *      token budgets B_i (Box 5, Eq. token_budget), the cosine threshold
 *      schedule with block end thresholds theta_e^(b) (Boxes 3-4), position
 *      thresholds (Box 6, Eqs. position_threshold and position_commit), the
 *      grinding detector and its force commit (Box 7, Eq. grinding-detector),
 *      all behind the model-adaptive gate (Section 4.6).
 *
 * Execution model.  Every call that takes a stream is asynchronous on that
 * stream (a CUDA stream handle, or NULL for the legacy default stream); the
 * library never synchronises the device on the step path.  The step kernels
 * use programmatic dependent launch: each may be scheduled while the kernel
 * before it in the stream still runs, and waits for that kernel to complete
 * before touching anything it produces (setting CAI_PDL=0 in the environment
 * before cai_init launches them plainly instead).  With B P <= 64 a step is
 * one kernel: the LM head over every row of the block, whose last CTA applies
 * the commit rule; it streams W before the previous step has committed and
 * waits for it only to write its partials and to commit (CAI_FUSED_MAX_BP=n
 * moves the limit, up to 256).  That LM head puts the rows in the MMA's A
 * operand and 256 vocabulary rows in N (up to 128 rows; CAI_ROWS_HEAD=0 uses
 * the swapped-operand kernel instead, W in A and the rows in N).  With B P > 64 a step is gather, LM head,
 * merge + commit.  The LM head is the CTA-pair
 * kernel (tcgen05 cta_group::2), which picks its orientation per step from
 * the masked-row count M: the rows as MMA N in row tiles of equal width (a
 * multiple of 32) while that width is at most 192, else as MMA M in 256-row
 * tiles.  A kernel that merges each row's per-tile partials follows it only
 * in contexts where some step size leaves more than one partial per pair and
 * CTA to merge.  CAI_PAIR_SWAP=0 keeps the pair kernel unswapped and moves
 * the steps below 32 rows to the single-CTA swapped-operand kernel (launched
 * on every step, returning at once on the others); CAI_PAIR_SWAP_MAX_N=n sets
 * the widest swapped tile; CAI_PAIR=0 runs every step on the single-CTA
 * kernel; CAI_PAIR_MIN_M=n sets the smallest step of the pair kernel (all
 * read at cai_init; CAI_NVTX=1 wraps every step call in an NVTX range).
 * cai_init_rmsnorm and CAI_DIAGNOSTICS
 * add one small kernel each to a single-kernel step.  The batch runs
 * blocks and steps in lockstep; sequences exit independently (Algorithm 1,
 * per sequence) and contribute no rows afterwards.  A context is not thread
 * safe; use one context per host thread.
 *
 * Status.  Every int-returning call returns CAI_OK (0) or a negative CAI_ERR_*
 * code; no C++ exception crosses the ABI.  After CAI_ERR_CUDA or
 * CAI_ERR_DEVICE the context is poisoned ("sticky"): every later call except
 * cai_free, cai_strerror and cai_device_error_bits returns the same code.
 */
#ifndef CAI_H
#define CAI_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ------------------------------------------------------------------ status */
#define CAI_OK 0
#define CAI_ERR_ARG (-1)         /* NULL pointer, bad enum, bad value            */
#define CAI_ERR_SHAPE (-2)       /* unsupported sizes (see cai_config)           */
#define CAI_ERR_ORDER (-3)       /* call out of order (see each step call)       */
#define CAI_ERR_CUDA (-4)        /* a CUDA runtime call failed (sticky)          */
#define CAI_ERR_TIMEOUT (-5)     /* cai_poll gave up waiting (not sticky)        */
#define CAI_ERR_DEVICE (-6)      /* a kernel's bounded wait gave up (sticky)     */
#define CAI_ERR_UNSUPPORTED (-7) /* the current device is not compute 10.3       */
#define CAI_ERR_NOMEM (-8)       /* an allocation failed                         */

/* ------------------------------------------------------------------- flags */
#define CAI_GATING 1u           /* Section 4.6 gate ON: budgets, grinding exit, force commit */
#define CAI_POS_FACTOR 2u       /* Box 6 position factors r_pos (else r = 1)                */
#define CAI_FLUSH_ON_EXIT 4u    /* commit still-masked tokens to their argmax when a block exits */
#define CAI_QUARTER_POS 8u      /* position/budget tiers at P/4, P/2, 3P/4 instead of 16/32/48 */
#define CAI_QUARTER_BLOCKS 16u  /* theta_e^(b) indexed by the quarter of the output block b is in */
#define CAI_NO_BLOCK_SCHEDULE 32u /* Box 3 alone: every block ends at theta_e1 (ablation "APD") */
#define CAI_FIXED_THRESHOLD 64u /* fixed-threshold rule (Fast-dLLM): theta^(b)(t) = theta_s      */
#define CAI_DIAGNOSTICS 128u    /* track stability steps t_i^* and drift D^(t) (Section 2.1)     */

#define CAI_PRESET_LLADA 0      /* gating ON  (Section 5: LLaDA-8B-Instruct) */
#define CAI_PRESET_DREAM 1      /* gating OFF (Section 5: Dream-7B-Instruct) */

#define CAI_MASK_TOKEN (-1)     /* token id of a still-masked position */

/* exit reasons of a block, per sequence (Algorithm 1) */
#define CAI_RUNNING 0
#define CAI_EXIT_DONE 1         /* no masked token remained                 */
#define CAI_EXIT_GRIND 2        /* grinding phase detected (Box 7)          */
#define CAI_EXIT_TMAX 3         /* reached local step T - 1                 */

/*
 * Workload and controller hyperparameters.  Algorithm 1 inputs: T, theta_s,
 * theta_e^(b) (via theta_e1 - theta_e_step (b - 1), floored at theta_e_min),
 * theta_fb, w (warmup_pct / 100), K, eta_bar.
 *
 * Shape limits (else CAI_ERR_SHAPE): B >= 1; 1 <= P <= 256; H % 64 == 0 and
 * 64 <= H <= 16384; V >= 64; 1 <= T <= 32767; 1 <= n_blocks <= 32767;
 * B * P <= 65536.
 */
typedef struct cai_config {
  int32_t B;           /* sequences in the batch                                  */
  int32_t P;           /* block length (positions per block)                      */
  int32_t H;           /* hidden size                                             */
  int32_t V;           /* vocabulary size                                         */
  int32_t T;           /* maximum denoising steps per block                       */
  int32_t n_blocks;    /* blocks per generation (generation length / P)           */
  double theta_s;      /* Box 3 start threshold, 0.90                             */
  double theta_e1;     /* Box 4 end threshold of block 1, 0.70                    */
  double theta_e_step; /* Box 4 decrease per block, 0.10                          */
  double theta_e_min;  /* floor of theta_e^(b) for b > 4, 0.40                     */
  int32_t warmup_pct;  /* Box 3 warm-up fraction w in percent, 15                 */
  int32_t K;           /* Box 7 patience window, 4                                */
  double theta_fb;     /* Box 7 force-commit threshold, 0.40                      */
  double clip_lo;      /* Box 6 clip range, 0.20                                  */
  double clip_hi;      /*                   0.98                                  */
  double eta_bar;      /* Box 7 low-yield threshold: 1.5 (count) or 0.015 (fraction) */
  int32_t eta_mode;    /* 0: eta counts new commits; 1: eta / (n_blocks P)        */
  uint32_t flags;      /* CAI_* flags above                                       */
} cai_config;

typedef struct cai_ctx cai_ctx;

/*
 * Device views of the controller state (all device pointers, owned by the
 * context, valid until cai_free).  L = n_blocks * P.  Row-major.
 */
typedef struct cai_state_view {
  int32_t* tok;         /* [B, L] committed token id, CAI_MASK_TOKEN while masked   */
  float* conf;          /* [B, L] c_i at the last step that saw the token masked    */
  float* s0;            /* [B, L] first-step confidence s_i (Box 2)                 */
  uint8_t* budget;      /* [B, L] B_i in {8, 32, 64} (Box 5), 0 before the block    */
  int16_t* cstep;       /* [B, L] local step at which the token committed, -1       */
  int32_t* cand;        /* [B, L] argmax at the last step that saw the token masked */
  int32_t* ell;         /* [B] low-yield counter of the current block (Algorithm 1) */
  int32_t* eta;         /* [B] tokens committed by the commit rule at the last step */
  int32_t* exit_reason; /* [B, n_blocks] CAI_RUNNING / CAI_EXIT_*                   */
  int32_t* exit_step;   /* [B, n_blocks] local step of the exit, -1                 */
  int32_t* unresolved;  /* [B, n_blocks] tokens left masked at the exit             */
  int32_t* m_hist;      /* [n_blocks, T] masked rows decoded by each step (M_t)     */
  /* CAI_DIAGNOSTICS (Section 2.1); left at their reset values otherwise: */
  uint8_t* run;         /* [B, L] consecutive decoded steps with the same argmax    */
  int16_t* stable;      /* [B, L] stability step t_i^*: the local step at which the
                           argmax has been the same for 3 consecutive decoded steps,
                           -1 until then (and for tokens committed earlier)        */
  float* drift;         /* [B, n_blocks, T] relative L2 drift D^(t) of the hidden
                           states between steps t-1 and t of a block, mean over
                           the block's P positions (Eq. relative_drift); NaN at
                           t = 0 and for steps not run                             */
} cai_state_view;

/*
 * Host copy of the controller state, for cai_state_download / cai_state_upload.
 * Each pointer is caller-owned host memory of the size given in
 * cai_state_view, or NULL to skip that field.  blk and t_next are the host
 * counters: the 0-based current block and the next local step to run.
 */
typedef struct cai_host_state {
  int32_t* tok;
  float* conf;
  float* s0;
  uint8_t* budget;
  int16_t* cstep;
  int32_t* cand;
  int32_t* ell;
  int32_t* eta;
  int32_t* exit_reason;
  int32_t* exit_step;
  int32_t* unresolved;
  int32_t* m_hist;
  uint8_t* run;
  int16_t* stable;
  float* drift;
  int32_t blk;
  int32_t t_next;
} cai_host_state;

/* Counters kept by the context (host side) since cai_init. */
typedef struct cai_stats {
  int64_t steps;            /* step calls issued                                   */
  int64_t launches;         /* kernels launched by this context                    */
  int64_t head_launches;    /* launches of the LM-head kernel                      */
  double head_ms;           /* summed device time of profiled LM-head launches     */
  int64_t head_profiled;    /* LM-head launches timed (cai_profile enabled)        */
  int32_t grid;             /* CTAs of the LM-head kernel                          */
  int32_t stages;           /* pipeline stages of the LM-head kernel               */
  int32_t n_max;            /* positions per MMA chunk (N of the swapped MMA)      */
  int32_t kernels_per_step; /* 1: single-kernel step (B P <= 64); else gather,
                               LM head(s), row merge if needed, commit (2 to 5)    */
  double step_ms;           /* summed device time of profiled steps, every kernel  */
  int32_t pair_grid;        /* CTAs of the CTA-pair LM head (0: not used)          */
  int32_t pair_swap_max_n;  /* steps whose tile width in the swapped orientation
                               (masked rows in the MMA N dimension) is at most
                               this run swapped on the pair LM head (0: never)     */
  int32_t pair_stages;      /* pipeline stages of the pair LM head                 */
  int32_t head_rows;        /* 1: single-kernel steps run the LM head with the rows
                               as the MMA's A operand (B P <= 128), 0: otherwise   */
} cai_stats;

/* Fill *cfg with the paper's hyperparameters (Section 5, Appendix "Setup")
 * for the given preset and shapes.  Returns CAI_ERR_ARG for a bad preset. */
int cai_config_default(cai_config* cfg, int32_t preset, int32_t B, int32_t P, int32_t H,
                       int32_t V, int32_t T, int32_t n_blocks);

/*
 * Create a context.  W is the LM-head weight [V, H] bf16, row-major, host or
 * device memory.  It is read once, during this call, into the library's
 * packed copies (2 V H bytes each: one copy when B P <= 64, two otherwise);
 * the caller may free or change it afterwards.  All state starts at block 0,
 * t = 0, every token masked.  Allocates device memory and one page of mapped
 * pinned host memory.  Synchronous.
 * Errors: CAI_ERR_ARG (NULL cfg/W/out), CAI_ERR_SHAPE, CAI_ERR_UNSUPPORTED,
 * CAI_ERR_NOMEM, CAI_ERR_CUDA.
 */
int cai_init(const cai_config* cfg, const void* W, void* stream, cai_ctx** out);

/*
 * cai_init with the model's final RMSNorm inside the decoding head.  The paper
 * has no counterpart: Box 1's p_theta is computed from the normalised last
 * hidden state, and this entry point lets the caller pass the last layer's
 * output before that norm, saving the pass over the hidden states that a
 * separate norm kernel would make.  Each decoded row h then becomes
 *   x = g * h / sqrt(mean_k h_k^2 + eps)
 * before z = W x.  norm_weight g is [H] bf16 (host or device; read during this
 * call only); eps >= 0.  The weight is folded into the library's packed copies
 * of W (W[v,k] g[k], rounded to bf16 once); 1 / sqrt(mean h^2 + eps) is
 * computed per row in fp32 from the bf16 row and scales the row's logits in
 * fp32 before the softmax.  Single-kernel steps add one small kernel per step
 * for the row scales; multi-kernel steps compute them in the gather.
 * Errors: as cai_init, and CAI_ERR_ARG for a NULL or misaligned norm_weight or
 * a negative or non-finite eps.
 */
int cai_init_rmsnorm(const cai_config* cfg, const void* W, const void* norm_weight, double eps,
                     void* stream, cai_ctx** out);

/*
 * Vocabulary-parallel decoding head.  Box 1's confidence and argmax are a
 * maximum, a sum of exponentials and a lowest-index argmax over the
 * vocabulary, and each of them is an exact merge of the same reductions over
 * the parts of any split of the vocabulary.  So g shards (one per GPU, or
 * several on one GPU) can each hold a slice of W and decode it: every shard
 * context keeps a full copy of the controller state, computes for every
 * masked row one triple over its slice, the triples of all shards are
 * exchanged (an all-gather of rows x 16 bytes per shard, by the caller:
 * torch.distributed, NCCL or anything else), and every shard merges them and
 * applies the same commit rule, so the states stay identical.
 *
 * cai_init_vocab_shard creates a shard context.  cfg->V is the size V of the
 * whole vocabulary; W_shard [V_shard, H] bf16 (row-major, host or device,
 * read during the call as for cai_init) holds its rows [v0, v0 + V_shard).
 * Requires 0 <= v0, V_shard >= 64 and v0 + V_shard <= V (else
 * CAI_ERR_SHAPE).  A shard context always runs multi-kernel steps; the plain
 * step calls refuse it (CAI_ERR_ARG).  A step is, in this order:
 *
 *   cai_shard_head(ctx, hidden, triples, stream): the gather, the shard's LM
 *   head and, into `triples` (device, 16-byte aligned, cai_shard_rows()
 *   entries of 16 bytes), one triple per row of the step's masked-row list:
 *   {float m = max z * log2(e), float S = sum 2^(z log2(e) - m), int32 idx
 *   = the lowest global vocabulary index reaching the maximum, 0}, the empty
 *   triple {-3e38, 0, INT32_MAX, 0} past the step's M rows.  Step zero of a
 *   block when the context's next local step is 0, else a denoising step,
 *   with the order rules of cai_first_step / cai_denoise_step; hidden as
 *   there (device, or page-locked host rows read in place by the gather).
 *
 *   cai_shard_commit(ctx, gathered, n_shards, stream): `gathered` (device,
 *   16-byte aligned) holds every shard's triples one after the other,
 *   [n_shards][cai_shard_rows()] (any order of shards: ties keep the lower
 *   index); merges each row's n_shards triples into c = 1 / S and the argmax
 *   and applies the commit rule, ending the step.  Errors: CAI_ERR_ORDER
 *   without a preceding cai_shard_head; CAI_ERR_ARG for n_shards outside
 *   [1, 4096] or a pointer that is not device memory.
 *
 * Between the two calls, cai_block_advance returns CAI_ERR_ORDER.  The
 * library performs no communication itself.
 */
int cai_init_vocab_shard(const cai_config* cfg, const void* W_shard, int32_t v0, int32_t V_shard,
                         void* stream, cai_ctx** out);
/* Rows of a shard context's exchange buffers (B P rounded up to 16). */
int cai_shard_rows(const cai_ctx* ctx, int32_t* rows);
int cai_shard_head(cai_ctx* ctx, const void* hidden, void* triples, void* stream);
int cai_shard_commit(cai_ctx* ctx, const void* gathered, int32_t n_shards, void* stream);

/*
 * Local step t = 0 of the current block (Algorithm 1, step-zero init): every
 * position of every sequence is masked, so M = B P rows are decoded.  Stores
 * s_i and B_i, then applies the commit rule with theta^(b)(0).
 * hidden: the block's final hidden states [B, P, H] bf16, row-major; row
 * (b, p) is the one that predicts position p of the block.  Device pointer:
 * read on the stream, must stay valid until the stream passes this call.
 * Host pointer: the rows are copied to the device on a stream of the
 * context's own into one of two alternating device buffers, which the step's
 * first kernel that reads them (the single-kernel LM head, or the gather)
 * waits for on the device, so the copy for the next step runs during this one
 * and the step's stream itself waits for nothing (with CAI_DIAGNOSTICS, or
 * the final norm in a single-kernel step, the step's stream waits for the
 * copy instead).  Page-locked memory must stay valid until the stream passes
 * this call; pageable memory is staged by the CUDA runtime before the call
 * returns.
 * Errors: CAI_ERR_ARG, CAI_ERR_ORDER (the block already ran a step; call
 * cai_block_advance or cai_reset first).
 */
int cai_first_step(cai_ctx* ctx, const void* hidden, void* stream);

/*
 * Local steps t = 1 .. T - 1 of the current block: decodes only the rows that
 * are still masked in sequences that have not exited; a step issued after all
 * sequences exited decodes nothing.  hidden as for cai_first_step.
 * Errors: CAI_ERR_ORDER before cai_first_step of the block, after T steps, or
 * after cai_poll has reported that every sequence exited the block.
 */
int cai_denoise_step(cai_ctx* ctx, const void* hidden, void* stream);

/*
 * Move to the next block (b += 1).  Host bookkeeping only; the low-yield
 * counters are reset by the next cai_first_step.  Sequences still running in
 * the old block keep CAI_RUNNING there.  Errors: CAI_ERR_ORDER if the current
 * block never ran a step or it is the last block.
 */
int cai_block_advance(cai_ctx* ctx, void* stream);

/* Start a new generation with the same weight: every token masked, block 0,
 * counters cleared.  Asynchronous on the stream (device memsets only). */
int cai_reset(cai_ctx* ctx, void* stream);

/*
 * Bounded host wait for the device's commit of the step issued `lag` step
 * calls ago (lag = 0: the last one), read from mapped pinned memory without a
 * device synchronisation.  On CAI_OK, *all_done is 1 if every sequence has
 * exited the current block as of that step (or a later one), else 0.
 * Errors: CAI_ERR_TIMEOUT after timeout_ms (not sticky); CAI_ERR_DEVICE if a
 * kernel reported a failed bounded wait; CAI_ERR_ARG for lag < 0.
 */
int cai_poll(cai_ctx* ctx, int32_t lag, int32_t timeout_ms, int32_t* all_done);

/* Device pointers of the state arrays (no copy, no synchronisation). */
int cai_get_state(cai_ctx* ctx, cai_state_view* out);

/* Synchronous copy of the whole state to caller host buffers (device
 * synchronise first), and back (checkpoint / resume, teacher forcing). */
int cai_state_download(cai_ctx* ctx, cai_host_state* dst);
int cai_state_upload(cai_ctx* ctx, const cai_host_state* src);

/* Asynchronous copy of the committed tokens [B, L] int32 into host memory on
 * the stream (pinned memory for a truly asynchronous copy). */
int cai_read_tokens(cai_ctx* ctx, int32_t* host_tokens, void* stream);

/* Time every step with CUDA events on its stream (enable = 1) or stop (0):
 * the LM-head launch(es) (head_ms) and the whole step (step_ms).  The events
 * sit between kernels, so profiled steps run without programmatic overlap.
 * cai_get_stats synchronises the events and reports the sums. */
int cai_profile(cai_ctx* ctx, int32_t enable);
int cai_get_stats(cai_ctx* ctx, cai_stats* out);

/* The context's device error word, which kernels set when a bounded wait
 * gives up (the reason behind CAI_ERR_DEVICE): one bit per kind of wait,
 * 0 while none has.  A synchronous copy (after the device's work so far);
 * also answers on a sticky context.  Errors: CAI_ERR_ARG, CAI_ERR_CUDA. */
#define CAI_DEVERR_WAIT_EMPTY     (1u << 0) /* producer waiting for a free stage          */
#define CAI_DEVERR_WAIT_FULL      (1u << 1) /* MMA issuer waiting for a loaded stage      */
#define CAI_DEVERR_WAIT_ACC_FULL  (1u << 2) /* epilogue waiting for an accumulator        */
#define CAI_DEVERR_WAIT_ACC_EMPTY (1u << 3) /* MMA issuer waiting for a drained accum.    */
#define CAI_DEVERR_DRAIN          (1u << 4) /* abort path draining copies in flight       */
#define CAI_DEVERR_BAD_ROW        (1u << 5) /* a masked token had no row in the list      */
#define CAI_DEVERR_WAIT_EPI       (1u << 6) /* epilogue warps waiting for each other      */
#define CAI_DEVERR_BOUNDS         (1u << 7) /* debug builds: index or offset out of range */
#define CAI_DEVERR_WAIT_ROWS      (1u << 8) /* staged host rows did not arrive            */
int cai_device_error_bits(cai_ctx* ctx, uint32_t* bits);

/* Release everything the context owns.  Synchronises the device first.
 * NULL is a no-op. */
void cai_free(cai_ctx* ctx);

/*
 * Decoding head over caller rows without allocating anything.  The paper has
 * no counterpart: this is a convenience for callers that cannot call
 * cudaMalloc where they need the head (a memory pool that owns the whole
 * device, an allocator-free runtime that reserved everything up front, a
 * region where an allocation would synchronise the device).  No context is
 * needed and nothing is allocated: no cudaMalloc, cudaFree or allocating
 * library call.
 *
 * For each of the M rows of `rows` ([M, H] bf16, device), computes
 * conf[i] = max_v softmax(W rows[i])_v and argmax[i] = the lowest v reaching
 * that maximum, against the caller's W ([V, H] bf16 row-major, device, read in
 * place).  conf (float) and argmax (int32) are device arrays of M entries.
 * Asynchronous on `stream`.  Limits: 1 <= M <= 256, V >= 128, H % 64 == 0 and
 * 64 <= H <= 16384 (else CAI_ERR_SHAPE); W and rows 16-byte aligned, and all
 * four pointers device (or managed) memory of the current device (else
 * CAI_ERR_ARG, with nothing launched).  Any CUDA error already pending from
 * earlier work is cleared first; if the LM-head kernel fails to launch, the
 * call returns CAI_ERR_CUDA without launching the merge.
 *
 * Scratch: a fixed file-scope device array of 256 x 160 partial triples
 * (640 KiB) plus an error word, held by every GPU that loads this library until
 * the process exits, shared by all calls and keeping the last call's
 * contents.  Calls that overlap on the GPU (on different streams, or from
 * different threads) race on it.  The first call on each device looks up the
 * array's device address and sets the kernel's shared-memory limit, with that
 * device current; make that first call before any stream capture.  If a
 * kernel-side bounded wait gives up, that call's outputs are NaN / -1.
 */
int cai_head_rows_static(const void* W, int32_t V, int32_t H, const void* rows, int32_t M,
                         float* conf, int32_t* argmax, void* stream);

/*
 * Testing hook for cai_head_rows_static: the next call (process-wide, once)
 * runs, between its LM-head and merge kernels, a kernel that waits through
 * the step kernels' bounded barrier wait on a barrier nothing arrives at and,
 * after the 2 s limit, records a failed wait in the static error word, as a
 * kernel whose wait gave up would.  That call's outputs are then NaN / -1 and
 * the word is cleared for the next call.  No trap and no fault.
 */
int cai_test_static_wait_timeout(void);

/* Static string for a status code. */
const char* cai_strerror(int status);

/*
 * Testing hook: make the n-th device allocation from now fail (n >= 1), as if
 * cudaMalloc had returned an error; n = 0 disables.  Process-wide.
 */
int cai_test_fail_alloc_after(int32_t n);

/*
 * Testing hook: cap the number of CTAs of the LM-head kernel for contexts
 * created from now on (n >= 1), so that small vocabularies still give each
 * CTA several 128-row tiles; n = 0 restores one CTA per SM.  Process-wide.
 */
int cai_test_head_grid_limit(int32_t n);

/*
 * Testing hook: every device buffer of a context is followed by 256 guard
 * bytes of a fixed pattern.  Synchronises the device, then sets *n_bad to the
 * number of buffers whose guard bytes changed (a write past their end).
 */
int cai_test_check_guards(cai_ctx* ctx, int32_t* n_bad);

/*
 * Testing hook: launches, on the stream, a kernel that waits through the
 * step kernels' bounded barrier wait on a barrier nothing arrives at; after
 * the wait limit (2 s) it records a wait failure in the context's error word
 * and returns.  The next call that reads the word (cai_poll,
 * cai_state_download) then returns CAI_ERR_DEVICE and the context is sticky.
 * No trap and no fault: the device and other contexts stay usable.
 */
int cai_test_wait_timeout(cai_ctx* ctx, void* stream);

/*
 * Testing hook, host only (no device use): the CTA-pair LM head's plan for a
 * step with M masked rows on n_pairs pairs whose widest swapped tile is
 * swap_max_n (0: never swapped).  Writes out[0] = 1 if the step runs in the
 * swapped orientation, out[1] = row tiles, out[2] = rows per row tile (the
 * MMA N when swapped, 256 otherwise), out[3] = partials per row read by the
 * commit (0: per-tile partials merged by the row-merge kernel).
 * CAI_ERR_ARG for M < 1, n_pairs < 1, swap_max_n < 0 or out == NULL.
 */
int cai_test_pair_plan(int32_t M, int32_t n_pairs, int32_t swap_max_n, int32_t* out);

/*
 * Testing hook, host only (no device use): the position thresholds
 * theta_i(t) (Box 6, Eq. position_threshold: the block threshold of Boxes 3
 * and 4 times the position factor, clipped to [clip_lo, clip_hi]) that a step
 * of block blk (0-based) at local step t hands to the commit rule, one fp32
 * value per position p < P into out[P].  Computed in double and rounded once,
 * exactly as for the step.  CAI_ERR_ARG for a null pointer, blk outside
 * [0, n_blocks) or t outside [0, T); otherwise cai_init's configuration checks.
 */
int cai_test_theta_table(const cai_config* cfg, int32_t blk, int32_t t, float* out);

#ifdef __cplusplus
}
#endif

#endif /* CAI_H */
