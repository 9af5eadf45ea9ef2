/*
 * CPU oracle for block-wise diffusion-LLM (LLaDA-style) decoding, as
 * described in "Efficient On-Device Diffusion LLM Inference with Mobile NPU"
 * (arXiv 2606.13740), Sec. 2.1 (block-wise decoding, prefix KV reuse) and
 * Sec. 3.2-3.3 (decoding window, draft tokens, staged stabilisation).
 *
 * TEST INFRASTRUCTURE ONLY.  This library is a plain, slow, obviously
 * correct restatement of what the GPU path computes.  Only the test suite,
 * the smoke check and the benchmark's CPU-baseline leg may load it.  It
 * shares no source with the CUDA library and includes none of its headers.
 *
 * Arithmetic: fp32 storage, fp64 accumulation in every dot product, softmax
 * sum and norm.  Weights are bf16 bit patterns widened exactly to fp32.
 */
#ifndef DLLM_ORACLE_H
#define DLLM_ORACLE_H
#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Token states (Sec. 3.3 "Staged Token Stabilization" plus the draft flag
 * of Sec. 3.2).  COMMITTED = visible but revisable; STABLE = long-term. */
enum { ORC_FIXED = 0, ORC_MASKED = 1, ORC_COMMITTED = 2, ORC_STABLE = 3, ORC_DRAFT = 4 };

/* Tensor ids used by the counter-based weight generator. */
enum { ORC_T_EMBED = 1, ORC_T_HEAD = 2 };
enum { ORC_W_Q = 0, ORC_W_K = 1, ORC_W_V = 2, ORC_W_O = 3, ORC_W_GATE = 4, ORC_W_UP = 5, ORC_W_DOWN = 6 };
#define ORC_LAYER_TENSOR(l, w) (16ull + 8ull * (uint64_t)(l) + (uint64_t)(w))
#define ORC_KV_TENSOR(b, l, c, L) (0x100000000ull + ((uint64_t)(b) * (uint64_t)(L) + (uint64_t)(l)) * 2ull + (uint64_t)(c))

typedef struct {
    int n_layers, d_model, n_heads, head_dim, ffn, vocab, mask_id;
    double rope_base, rms_eps;
    uint64_t weight_seed;
    /* K/V heads (grouped-query attention, as in the Dream-7B model of Sec. 5.1); 0 = n_heads
     * (multi-head attention, LLaDA).  Must divide n_heads: query head h reads K/V head
     * h / (n_heads / n_kv_heads). */
    int n_kv_heads;
    /* Storage of the projection weights (the seven per layer and the LM head; the embedding is
     * always bf16): 16 (or 0) = bf16 drawn N(0, 0.02); 4 = the 4-bit block format of the Q4_0
     * weights the paper runs (Sec. 5.1), see orc_q4_dequant.  The oracle keeps every weight as
     * the bf16 value it dequantizes to, so the arithmetic after it is the same for both. */
    int weight_bits;
} orc_config;

typedef struct {
    int steps_per_block;   /* S */
    int block_len;         /* 32 */
    float theta_remask;    /* 0 disables the revision pass */
    float theta_stable;    /* promotion to STABLE */
    int remask_max;        /* R_max re-masks per step */
    int spec_trigger;      /* lookahead when masked count <= trigger */
    int spec_blocks;       /* future blocks added to the window; 0 = off */
    int use_prefix_cache;  /* 0 = vanilla full-sequence decoding */
    int commit_mode;       /* ORC_COMMIT_SCHEDULE or ORC_COMMIT_THRESHOLD */
    float theta_visible;   /* threshold mode: promotion of a masked position to visible */
    int scr_rows;          /* sparse cache refresh: prefix positions re-scored per step (0 = off) */
    /* Adaptive lookahead (Sec. 3.2): with spec_allowance >= 0 and a latency table, the window
     * takes the largest k <= spec_blocks future blocks for which every step up to k stays
     * within (1 + spec_allowance) times the latency without lookahead: spec_lat[i] = the step
     * latency with a window of i + 1 blocks.  spec_allowance < 0: all spec_blocks (fixed). */
    float spec_allowance;
    int spec_lat_n;
    float spec_lat[8];
    /* Continuous sliding (Sec. 3.2, with the prefix cache): the window keeps the size of a block
     * (plus lookahead blocks) and starts at the cache frontier kv_len.  After the commit pass the
     * longest leading run of window positions that were visible (COMMITTED or STABLE) when the
     * forward ran and still are joins the prefix cache with the K/V that forward computed for
     * them, so the window slides right into the next block, whose positions it drafts like
     * lookahead blocks.  Positions that left the window are no longer revised. */
    int slide;
} orc_sched;

/* Commit rules.  SCHEDULE: LLaDA's fixed schedule, ceil(m / (S - step)) of the m masked
 * positions per step, the most confident first.  THRESHOLD: staged token stabilization
 * (Sec. 3.3): every masked position whose confidence reaches theta_visible becomes visible
 * (COMMITTED), STABLE if it also reaches theta_stable; when none reaches theta_visible, the
 * single most confident one becomes visible, so every step makes progress. */
enum { ORC_COMMIT_SCHEDULE = 0, ORC_COMMIT_THRESHOLD = 1 };

typedef struct {
    int n_committed, n_remasked, n_stable, n_drafts, block_done, masked_after;
    int n_refreshed, n_revised;  /* sparse cache refresh: prefix K/V rows merged, prefix ids revised */
} orc_step_out;

/* Sparse cache refresh (Sec. 3.3, with the prefix cache on): each step the first scr_rows
 * prefix positions (ascending) in the visible state (COMMITTED) ride along with the window as
 * extra query rows at their own positions; they attend to the cached prefix as it stands and
 * to the window, and add no keys.  After the window's commit pass each of them is re-scored:
 * at tokconf >= theta_stable it becomes STABLE; below theta_remask (when > 0) with an argmax
 * other than its id it takes that argmax; otherwise it keeps its id.  Every one that keeps its
 * id has the K/V computed for it this step written into the cache at its position (the merge
 * happens at the step boundary: nothing of it is visible inside the step). */

/* ---- counter-based generator (SplitMix64, Steele/Lea/Flood 2014) ---- */
uint64_t orc_splitmix_at(uint64_t key, uint64_t n);
void orc_gen_f32(uint64_t seed, uint64_t tensor_id, uint64_t first, uint64_t n, double sigma, float* out);
void orc_gen_bf16(uint64_t seed, uint64_t tensor_id, uint64_t first, uint64_t n, double sigma, uint16_t* out);
uint16_t orc_f32_to_bf16(float f);
float orc_bf16_to_f32(uint16_t h);

/* ---- 4-bit block-quantised weights (Q4_0, Sec. 5.1) ----
 * Along the input dimension every 32 consecutive weights of a row form a block with one scale
 * d; each weight is a 4-bit code q in 0..15 and stands for d * (q - 8).  The paper's Q4_0 keeps
 * d in fp16; here d is a bf16 value (reading: the GPU multiplies in bf16), and the weight the
 * arithmetic uses is d * (q - 8) rounded once to bf16 (the product itself is exact in fp32).
 * Synthetic draws (no trained weights): for tensor tid, q of element (r, c) = the top 4 bits
 * of SplitMix64 output r*cols + c of the stream keyed by (seed, ORC_Q4_CODES + tid); d of
 * block (r, b) = the bf16 with bits 0x3B80 | (top 5 bits of output r*ceil(cols/32) + b of the
 * stream keyed by (seed, ORC_Q4_SCALES + tid)), i.e. (1 + m/128) * 2^-8, m in 0..31: the
 * weights' standard deviation is then about 0.02, that of the bf16 weights N(0, 0.02). */
#define ORC_Q4_CODES (3ull << 40)
#define ORC_Q4_SCALES (4ull << 40)
uint16_t orc_q4_dequant(int code, uint16_t scale_bits);
int orc_q4_code(uint64_t seed, uint64_t tid, int cols, int r, int c);
uint16_t orc_q4_scale(uint64_t seed, uint64_t tid, int cols, int r, int b);
/* rows x cols weights of tensor tid in the 4-bit format, dequantised to bf16 bits. */
void orc_gen_q4(uint64_t seed, uint64_t tid, int rows, int cols, uint16_t* out);

/* ---- model ---- */
typedef struct orc_model orc_model;
/* gen_layers < 0: all layers; gen_head: generate the LM head. */
orc_model* orc_model_new(const orc_config* c, int gen_layers, int gen_head);
orc_model* orc_model_new_zero(const orc_config* c);
/* Direct access to a weight (bf16 bits, logical row-major [out][in]).
 * layer = -1: which = ORC_T_EMBED / ORC_T_HEAD. */
uint16_t* orc_model_weight(orc_model* m, int layer, int which, size_t* n_elems);
float* orc_model_norm(orc_model* m, int layer, int which /*0 attn,1 ffn; layer -1: final*/);
void orc_model_free(orc_model* m);

/* ---- single ops (Sec. 2.1 transformer step), exposed for pins ---- */
void orc_rmsnorm(int n, const float* x, const float* gamma, double eps, float* out);
void orc_rope(int hd, double base, int pos, float* vec /* [hd], in place */);
/* logits -> decision (argmax excluding mask, max-softmax confidence). */
void orc_decide(int V, int mask_id, const float* logits, int32_t cur_tok,
                int32_t* x0, float* conf, float* tokconf, float* margin);

/* Forward over a window of T tokens at absolute positions pos[], against a
 * prefix of P cached keys/values per layer (prefix_k/v: [L][P][d], NULL if
 * P == 0).  group (nullable): window key j is visible to window query i iff
 * group[j] <= group[i].  out_k/out_v (nullable): window K/V [L][T][d].
 * logits (nullable): [T][V]; head skipped when NULL.  Returns 0. */
int orc_forward(const orc_model* m, int T, const int32_t* tok, const int32_t* pos,
                int P, const float* prefix_k, const float* prefix_v, const int32_t* group,
                float* out_k, float* out_v, float* logits, int n_layers_run);
/* The same with only the first Tk of the T rows as keys (the rest are queries only). */
int orc_forward_ex(const orc_model* m, int T, int Tk, const int32_t* tok, const int32_t* pos,
                   int P, const float* prefix_k, const float* prefix_v, const int32_t* group,
                   float* out_k, float* out_v, float* logits, int n_layers_run);

/* One commit / re-mask / draft pass (C5-C9 of the scope table) over a
 * single sequence's state arrays (length n_pos).  Pure function. */
int orc_commit(const orc_sched* s, int mask_id, int n_pos, int32_t* tok, uint8_t* st,
               int w0, int T, int c0, int c1, int step, const int32_t* x0, const float* conf,
               const float* tokconf, orc_step_out* out);

/* ---- stateful session (one sequence) ---- */
typedef struct orc_session orc_session;
orc_session* orc_session_new(const orc_model* m, const orc_sched* s, int Lp, const int32_t* prompt, int gen_len);
void orc_session_free(orc_session* x);
/* The last step's tracked prefix positions (sparse cache refresh) and their decisions (arrays
 * of scr_rows entries, nullable); returns how many there were. */
int orc_scr_decisions(const orc_session* x, int32_t* pos, int32_t* x0, float* conf, float* tokconf, float* margin);
int orc_prefill(orc_session* x);
/* 0: started a block; 1: generation finished (last block appended). */
int orc_begin_block(orc_session* x);
int orc_denoise_step(orc_session* x, orc_step_out* out, int keep_logits);
int orc_window(const orc_session* x, int32_t* info /* w0, T, c0, c1, step, kv_len, spec_on */);
int orc_step_decisions(const orc_session* x, int32_t* x0, float* conf, float* tokconf, float* margin, float* logits);
int orc_get_state(const orc_session* x, int32_t* tok, uint8_t* st, int32_t* kv_len);
int orc_set_state(orc_session* x, const int32_t* tok, const uint8_t* st);
/* prefix K/V of layer l: [kv_len][d] (pointer into the session). */
const float* orc_prefix_kv(const orc_session* x, int layer, int which);
int orc_n_pos(const orc_session* x);

#ifdef __cplusplus
}
#endif
#endif
