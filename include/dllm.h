/*
 * dllm.h - C ABI of the GB300 block-wise diffusion-LLM denoising path.
 *
 * Implements the decoding loop of "Efficient On-Device Diffusion LLM Inference
 * with Mobile NPU" (arXiv 2606.13740): block-wise decoding with prefix KV
 * reuse (Sec. 2.1 "Block-Wise Decoding"), the decoding window with draft
 * tokens from future blocks (Sec. 3.2 "Multi-Block Speculative Decoding"),
 * and revisable commits (Sec. 3.3 "Staged Token Stabilization").  Every step
 * of the path (embedding, RMSNorm, QKV+RoPE, attention, SwiGLU MLP, LM head
 * with confidence and argmax, commit/re-mask/draft) runs in the library's own
 * CUDA kernels on one GPU; there is no CPU fallback.
 *
 * Conventions for every entry point:
 *   - Return 0 (DLLM_OK) or a negative DLLM_E* code (DLLM_DONE = 1 is a
 *     non-error status of dllm_begin_block).  No C++ exception crosses the ABI.
 *   - Argument and capacity errors (DLLM_EINVAL, DLLM_ECAPACITY) are
 *     detected on the host; they leave the context usable (a request whose
 *     start failed is not started: call dllm_prefill again).  Every other error (DLLM_ENOMEM, DLLM_ECUDA,
 *     DLLM_ETIMEOUT, DLLM_ESTATE from a failed generation) poisons the
 *     context: later calls return DLLM_ESTATE until dllm_free.
 *     dllm_last_error gives the message of the last error.
 *   - Host pointers belong to the caller and are only read/written during the
 *     call.  Device memory belongs to the context (or to the caller's arena,
 *     which the context never frees).
 *   - Work is queued on the context's stream.  Calls that return host data
 *     synchronise that stream; the others are asynchronous.
 *   - Token ids are int32; token states are uint8 DLLM_FIXED..DLLM_DRAFT.
 *   - Sequences of a batch are independent and advance in lockstep (same
 *     prompt length, same block schedule).
 */
#ifndef DLLM_H
#define DLLM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define DLLM_OK 0
#define DLLM_DONE 1
#define DLLM_EINVAL (-1)
#define DLLM_ENOMEM (-2)
#define DLLM_ECUDA (-3)
#define DLLM_ETIMEOUT (-4)
#define DLLM_ESTATE (-5)
#define DLLM_ECAPACITY (-6)

/* Token states.  COMMITTED is the paper's "visible" state (usable as
 * context, still revisable); STABLE is long-term (Sec. 3.3); DRAFT marks a
 * future-block prediction (Sec. 3.2). */
enum { DLLM_FIXED = 0, DLLM_MASKED = 1, DLLM_COMMITTED = 2, DLLM_STABLE = 3, DLLM_DRAFT = 4 };

typedef struct dllm_ctx dllm_ctx;

/* Model shape and capacities.  The model is the LLaDA architecture the paper
 * runs (Sec. 5.1 "Models"): pre-norm RMSNorm, multi-head attention without a
 * causal mask, rotate-half RoPE, SwiGLU MLP, untied LM head.  Weights are
 * bf16, drawn on the device from weight_seed (N(0, 0.02) by a counter-based
 * SplitMix64/Irwin-Hall generator); RMSNorm gains are one.
 * n_kv_heads < n_heads gives grouped-query attention (the Dream-7B model the
 * paper also runs, Sec. 5.1): query head h reads K/V head h / (n_heads /
 * n_kv_heads), and the KV cache holds n_kv_heads heads.
 * Constraints: head_dim in {64, 128}; d_model, n_heads*head_dim multiples of
 * 128; n_kv_heads 0 (= n_heads) or a divisor of n_heads with
 * n_kv_heads*head_dim a multiple of 128; vocab, ffn multiples of 8;
 * max_window * max_batch <= 4096. */
typedef struct {
    int n_layers, d_model, n_heads, head_dim, ffn, vocab, mask_id;
    float rope_base, rms_eps;
    int max_batch;   /* sequences per call */
    int max_ctx;     /* positions per sequence: prompt + generation (+ window overhang) */
    int max_window;  /* query tokens per sequence per forward (window or prompt) */
    int block_len;   /* tokens per block (32) */
    uint64_t weight_seed;
    int n_kv_heads;  /* K/V heads; 0 = n_heads (multi-head attention, LLaDA) */
    /* Projection weights (the seven per layer and the LM head; the embedding is always bf16):
     * 16 (or 0): bf16; 4: the 4-bit block format of the Q4_0 weights the paper runs (Sec. 5.1):
     * 32 consecutive weights of a row (along the input dimension) share one bf16 scale d, each
     * weight is a 4-bit code q standing for d * (q - 8), and the tensor cores multiply the bf16
     * value of d * (q - 8) (rounded once); 4.5 bits per weight in HBM.  Drawn from weight_seed:
     * codes uniform over 0..15, scales (1 + m/128) * 2^-8 with m in 0..31 (standard deviation
     * of the weights about 0.02, as for the bf16 draws). */
    int weight_bits;
} dllm_config;

/* Commit rules (dllm_sched.commit_mode). */
enum { DLLM_COMMIT_SCHEDULE = 0, DLLM_COMMIT_THRESHOLD = 1 };

/* Decoding schedule.  steps_per_block = S.  commit_mode DLLM_COMMIT_SCHEDULE
 * (LLaDA's fixed schedule): the step-s commit count is ceil(m / (S - s)) for
 * m masked positions of the current block, the most confident first.
 * DLLM_COMMIT_THRESHOLD (staged token stabilization, Sec. 3.3): every masked
 * position whose confidence reaches theta_visible becomes COMMITTED (visible),
 * STABLE if it also reaches theta_stable; when none reaches theta_visible the
 * single most confident one becomes COMMITTED, so a block takes between 1 and
 * block_len steps (plus re-masks); S is then only the revision horizon.
 * theta_remask > 0 enables the revision pass: committed tokens whose
 * current-id probability is >= theta_stable become STABLE, and at most
 * remask_max of those below theta_remask (lowest first) are re-masked; it is
 * skipped on the block's last step.  spec_blocks > 0 enables lookahead: when
 * the current block has <= spec_trigger masked positions, the window extends
 * over the next spec_blocks blocks, each of which drafts its most confident
 * masked position per step.  use_prefix_cache = 0 gives vanilla decoding:
 * every step runs the full sequence and nothing is cached. */
typedef struct {
    int steps_per_block;
    float theta_remask;
    float theta_stable;
    int remask_max;
    int spec_trigger;
    int spec_blocks;
    int use_prefix_cache;
    int commit_mode;      /* DLLM_COMMIT_SCHEDULE or DLLM_COMMIT_THRESHOLD */
    float theta_visible;  /* threshold mode only */
    /* Sparse cache refresh (Sec. 3.3; with the prefix cache on; 0 = off, at most
     * DLLM_MAX_SCR_ROWS): each step, per sequence, the first scr_rows prefix positions that are COMMITTED
     * (visible, not stable) run with the window as extra query rows at their own positions,
     * attending to the prefix as cached and to the window and adding no keys.  After the
     * commit pass each is re-scored: STABLE at tokconf >= theta_stable; below theta_remask
     * (when > 0) with another argmax it takes that argmax; otherwise it keeps its id.  The K/V
     * computed for the rows that keep their id replace theirs in the prefix cache after the
     * step (the merge is not visible inside the step).  The window then counts scr_rows more
     * rows against max_window. */
    int scr_rows;
    /* Adaptive lookahead (Sec. 3.2): with spec_allowance >= 0 and spec_lat_n > 0, once the
     * lookahead triggers the window takes the largest k <= spec_blocks future blocks for which
     * every step up to k stays within (1 + spec_allowance) times the latency without lookahead;
     * spec_lat[i] = the measured step latency with a window of i + 1 blocks (the window-size
     * sweep).  k = 0 runs the plain window.  spec_allowance < 0: all spec_blocks (fixed). */
    float spec_allowance;
    int spec_lat_n;
    float spec_lat[8];
    /* Selective logits skipping (Sec. 3.3; 0 = off, 1 = on): the LM head, its softmax
     * statistics and the decision run only for the rows that still need one (positions that
     * are MASKED, COMMITTED or DRAFT, and refresh rows); FIXED and STABLE rows are skipped and
     * their step decisions read x0 = -1, conf = tokconf = 0.  Ignored while the logits are
     * captured for debugging. */
    int sls;
    /* Continuous sliding (Sec. 3.2; 0 = off, 1 = on; prefix cache on, batch 1): the window
     * keeps one block's length (plus lookahead blocks) and starts at the cache frontier; after
     * each step the leading run of window positions that were visible (COMMITTED or STABLE) at
     * the forward and still are joins the prefix cache with the K/V that forward computed, so
     * the window slides into the next block, drafting there as lookahead does.  Positions that
     * left the window are not revised; the block end appends only what has not slid. */
    int slide;
} dllm_sched;
#define DLLM_MAX_SCR_ROWS 32

/* Result of one denoising step, summed over the batch (block_done: all). */
typedef struct {
    int n_committed, n_remasked, n_stable, n_drafts, block_done, masked_after;
    int n_refreshed, n_revised;  /* sparse cache refresh: prefix K/V rows merged, prefix ids revised */
} dllm_step_out;

typedef struct {
    int steps;        /* denoising steps run */
    int spec_steps;   /* steps whose window included draft blocks */
    int blocks;       /* blocks finished */
} dllm_stats;

/* Device bytes the context needs for cfg (weights, KV cache, activations,
 * scratch).  Pass an arena of at least this size to dllm_init, or NULL. */
int dllm_arena_bytes(const dllm_config* cfg, size_t* bytes);

/* Create a context on the current CUDA device.  dev_arena: caller-owned
 * device memory of arena_bytes (>= dllm_arena_bytes), or NULL to let the
 * library allocate (and later free) its own.  cuda_stream: a cudaStream_t
 * (as void*), or NULL for a library-created stream.  Draws all weights.
 * Errors: DLLM_EINVAL (bad shape), DLLM_ENOMEM, DLLM_ECUDA. */
int dllm_init(const dllm_config* cfg, void* dev_arena, size_t arena_bytes, void* cuda_stream, dllm_ctx** out);

/* Free the context and everything it allocated (not a caller arena). */
void dllm_free(dllm_ctx* ctx);

/* Last error message of the context (static storage for a NULL ctx). */
const char* dllm_last_error(const dllm_ctx* ctx);

/* Wait for the context's stream and report device-side errors (a bounded
 * wait that ran out gives DLLM_ETIMEOUT). */
int dllm_sync(dllm_ctx* ctx);

/* Start a request (Sec. 2.1): batch sequences, prompt = host int32
 * [batch][Lp], gen_len masked positions after it.  With the prefix cache on,
 * runs the prompt through the layers (bidirectional over the prompt) and
 * stores its K/V as the prefix.  Errors: DLLM_EINVAL, DLLM_ECAPACITY
 * (Lp + gen_len + window overhang > max_ctx, batch > max_batch). */
int dllm_prefill(dllm_ctx* ctx, const dllm_sched* sched, int batch, const int32_t* prompt, int Lp, int gen_len);

/* Synthetic prefix instead of a prefill: every sequence gets P cached
 * positions whose K/V are drawn from seed (N(0,1), same generator), ids 0 and
 * state FIXED, followed by gen_len masked positions. */
int dllm_set_prefix_kv_random(dllm_ctx* ctx, const dllm_sched* sched, int batch, int P, int gen_len, uint64_t seed);

/* Advance to the next block (Sec. 2.1 "Block-Wise Decoding": blocks are
 * decoded left to right and a finished block's KV joins the reusable prefix;
 * Sec. 3.2: drafts a future block already holds are re-checked once it becomes
 * current).  If a block is current it must be finished (no
 * MASKED position, else DLLM_EINVAL); with the prefix cache on its K/V are
 * recomputed from its final ids (attending to prefix + block) and appended.
 * Drafts of the new block become COMMITTED (re-checked by the revision
 * pass).  Returns DLLM_DONE when no block is left. */
int dllm_begin_block(dllm_ctx* ctx);

/* One denoising step on the current window (Sec. 2.1 "Diffusion Large
 * Language Model": every unresolved position is predicted in parallel and a
 * confidence-selected subset is committed; Sec. 3.2: the window may extend
 * over future blocks, whose predictions become drafts; Sec. 3.3: committed
 * tokens are revised until stable): forward, decisions, commit / re-mask /
 * drafts.  out (nullable, host): filled after a stream sync; with
 * NULL the call stays asynchronous unless lookahead needs the masked count. */
int dllm_denoise_step(dllm_ctx* ctx, dllm_step_out* out);

/* Restore the request state to what it was at the last dllm_begin_block or
 * dllm_set_state, and reset the block's step counter (repeats identical
 * steps). */
int dllm_rewind_block(dllm_ctx* ctx);

/* Whole request (Sec. 2.1, the block-wise decoding loop with prefix KV
 * reuse; Sec. 3.2 / 3.3 as selected by sched): prefill, then blocks until
 * done.  out_tokens: host int32
 * [batch][gen_len].  stats nullable. */
int dllm_generate(dllm_ctx* ctx, const dllm_sched* sched, int batch, const int32_t* prompt, int Lp, int gen_len,
                  int32_t* out_tokens, dllm_stats* stats);

/* Current window (sequence 0): info[0..6] = w0, T, c0, c1, step, kv_len,
 * spec_on of the last step (positions absolute within the sequence). */
int dllm_window(dllm_ctx* ctx, int32_t* info);

/* Copy the whole state out: tokens int32 [batch][n_pos], states uint8
 * [batch][n_pos], kv_len int32 [batch] (any may be NULL).  Synchronises. */
int dllm_get_state(dllm_ctx* ctx, int32_t* tokens, uint8_t* status, int32_t* kv_len);

/* Overwrite tokens/states [batch][n_pos] (teacher forcing; either may be
 * NULL).  Inside a block this also becomes the dllm_rewind_block point. */
int dllm_set_state(dllm_ctx* ctx, const int32_t* tokens, const uint8_t* status);

/* Debug output of the last step, window-indexed [batch][T]: argmax ids,
 * max-softmax confidence, probability of the current id; logits fp32
 * [batch][T][vocab] only when dllm_set_debug enabled them (else pass NULL).
 * Synchronises. */
int dllm_get_step_debug(dllm_ctx* ctx, float* logits, int32_t* argmax, float* conf, float* tokconf);

/* The last step's sparse-cache-refresh rows: pos, argmax, conf, tokconf (host arrays
 * [batch][scr_rows], nullable; pos -1 = an unused row); *n = scr_rows.  Synchronises. */
int dllm_get_scr_debug(dllm_ctx* ctx, int32_t* pos, int32_t* argmax, float* conf, float* tokconf, int* n);

/* flags bit 0: materialise logits; bit 1: disable CUDA graphs; bit 2: launch
 * without programmatic dependent launch; bit 3: give the weight-streaming
 * projections 227 KB of shared memory (one CTA per SM, the deepest weight
 * ring) instead of leaving room beside them for the attention kernel's CTAs
 * (146 KB for the chained projections, 113 KB for dllm_op_gemm_*); bit 4:
 * record GEMM and attention timelines (dllm_get_trace); bit 5: the bounded-
 * wait test: the next denoising step's first projection waits for a device
 * word that nothing writes, so that wait runs out (after about 2 s) and the
 * step reports DLLM_ETIMEOUT, which poisons the context.  Bits 2 and 3 apply
 * process-wide (for A/B measurements). */
int dllm_set_debug(dllm_ctx* ctx, int flags);

/* Copy one weight back in its logical row-major layout (bf16 bits):
 * layer -1 with which 1 = embedding, 2 = LM head; otherwise which =
 * 0 q, 1 k, 2 v, 3 o, 4 gate, 5 up, 6 down.  Synchronises. */
int dllm_get_weight(dllm_ctx* ctx, int layer, int which, uint16_t* out, size_t n_elems);

/* Copy a slice of the K or V cache (which 0/1) of one layer and sequence:
 * out fp32 [n][n_kv_heads*head_dim] for positions [p0, p0+n).  Synchronises. */
int dllm_get_kv(dllm_ctx* ctx, int layer, int which, int seq, int p0, int n, float* out);

/* Kernel kinds of one denoising step, for dllm_get_profile. */
enum {
    DLLM_K_EMBED = 0,       /* embedding gather + first RMSNorm */
    DLLM_K_NORM = 1,        /* RMSNorm */
    DLLM_K_QKV = 2,         /* QKV projection + RoPE + window K/V write */
    DLLM_K_ATTN = 3,        /* attention (+ split combine) */
    DLLM_K_OPROJ = 4,       /* output projection + residual */
    DLLM_K_GATEUP = 5,      /* gate/up projection + SwiGLU */
    DLLM_K_DOWN = 6,        /* down projection + residual */
    DLLM_K_HEAD = 7,        /* LM head + per-tile softmax statistics */
    DLLM_K_HEAD_REDUCE = 8, /* current-id gather, vocab-tile merge */
    DLLM_K_COMMIT = 9,      /* commit / re-mask / drafts */
    DLLM_K_LAYER = 10,      /* chained projections of one layer: output (+ residual),
                               gate/up (+ SwiGLU), down (+ residual), then the next
                               layer's QKV or the LM head */
    DLLM_NKINDS = 11
};

/* Per-kernel timing of denoising steps: with enable, every launch of a step
 * is followed by a CUDA event on the context's stream (captured into the
 * step's graph) and each step synchronises to accumulate the elapsed time
 * between consecutive events by kind.  Enabling resets the totals. */
int dllm_set_profile(dllm_ctx* ctx, int enable);

/* Totals since dllm_set_profile(1): ms_total[DLLM_NKINDS] milliseconds,
 * launches_per_step[DLLM_NKINDS] launches of each kind in the last step,
 * steps profiled (any pointer may be NULL). */
int dllm_get_profile(dllm_ctx* ctx, double* ms_total, int32_t* launches_per_step, int32_t* steps);

/* With dllm_set_debug(16): per-CTA timelines (%globaltimer stamps) of the
 * GEMM and attention launches of the last step, in launch order: out
 * [n_launches][256][16].  GEMM slots as in dllm_op_gemm_trace; attention
 * slots 0 start, 1 dependency wait passed, 2 key loop done, 3 split ticket
 * taken, 4 merge done (last split only), 5 SM id, 6 last split.
 * Synchronises. */
int dllm_get_trace(dllm_ctx* ctx, unsigned long long* out, int max_launches, int32_t* n_launches);

/* Kernel launches in the last denoising step (all kinds). */
int dllm_launches_per_step(dllm_ctx* ctx, int32_t* n);

#ifdef __cplusplus
}
#endif
#endif
