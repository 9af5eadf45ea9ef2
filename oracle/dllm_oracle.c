/*
 * CPU oracle for block-wise diffusion-LLM (LLaDA-style) decoding,
 * arXiv 2606.13740 ("llada.cpp").
 *
 * TEST INFRASTRUCTURE ONLY: loaded by the test suite, the smoke check and
 * the benchmark's CPU-baseline leg, never by the product path.  It shares no
 * source, header, table or helper with the CUDA library.
 *
 * What it computes, and where the paper says so:
 *   - Sec. 2.1 "Diffusion Large Language Model": each denoising step predicts
 *     every unresolved position in parallel and commits a confidence-selected
 *     subset (orc_decide, orc_commit).
 *   - Sec. 2.1 "Block-Wise Decoding": blocks decoded left to right, the KV of
 *     completed blocks reused as a prefix (orc_begin_block, orc_prefill).
 *   - Sec. 3.2 "Multi-Block Speculative Decoding": a decoding window that may
 *     extend past the current block; future-block tokens are drafts that never
 *     update the prefix KV nor the commit order, and are re-checked when their
 *     block becomes current (orc_denoise_step, orc_commit).
 *   - Sec. 3.3 "Staged Token Stabilization": committed tokens stay revisable
 *     until a stability threshold is met (revision pass in orc_commit).
 *   - The transformer itself is the LLaDA architecture the paper runs
 *     (Sec. 5.1 "Models"): pre-norm RMSNorm, multi-head attention without a
 *     causal mask, rotate-half RoPE, SwiGLU MLP, untied LM head.
 *
 * Precision: fp32 storage, fp64 accumulation (dot products, softmax sums,
 * RMS).  Weights are bf16 bit patterns widened exactly to fp32.
 *
 * Parity pins (tests/test_oracle_*.py): brute-force and library checks of
 * every op on tiny shapes, softmax normalisation, RoPE as complex rotation,
 * exact commit counts, mask never committed, vanilla LLaDA equivalence,
 * incremental prefix KV == block-causal recomputation.
 */
#include "dllm_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ------------------------------------------------------------------ */
/* Counter-based generator: SplitMix64 (Steele, Lea & Flood, OOPSLA 2014). */
/* The n-th output of a stream whose state starts at `key` is               */
/* mix(key + (n+1) * golden_gamma).                                          */
/* ------------------------------------------------------------------ */
static uint64_t sm64_mix(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

uint64_t orc_splitmix_at(uint64_t key, uint64_t n) {
    return sm64_mix(key + (n + 1ull) * 0x9E3779B97F4A7C15ull);
}

/* Element i of tensor t: sum of four 32-bit draws (Irwin-Hall of order 4),
 * centred and scaled to unit variance, times sigma.  Every step is an exact
 * integer op or one correctly rounded IEEE double op, so any conforming
 * implementation of this definition reproduces the same float. */
static float gen_one(uint64_t key, uint64_t i, double sigma) {
    uint64_t s = 0;
    for (uint64_t j = 0; j < 4; ++j) s += orc_splitmix_at(key, 4ull * i + j) >> 32;
    double centred = (double)s - 8589934592.0; /* 2^33, exact */
    double unit = centred * 0x1.bb67ae8584caap-32; /* sqrt(3) / 2^32, one rounding */
    double scaled = unit * sigma;                  /* one rounding */
    return (float)scaled;
}

void orc_gen_f32(uint64_t seed, uint64_t tid, uint64_t first, uint64_t n, double sigma, float* out) {
    uint64_t key = orc_splitmix_at(seed, tid);
#pragma omp parallel for schedule(static)
    for (long long i = 0; i < (long long)n; ++i) out[i] = gen_one(key, first + (uint64_t)i, sigma);
}

uint16_t orc_f32_to_bf16(float f) {
    uint32_t b;
    memcpy(&b, &f, 4);
    if ((b & 0x7F800000u) == 0x7F800000u && (b & 0x007FFFFFu)) return 0x7FC0; /* NaN */
    uint32_t lsb = (b >> 16) & 1u;
    b += 0x7FFFu + lsb; /* round to nearest, ties to even */
    return (uint16_t)(b >> 16);
}

float orc_bf16_to_f32(uint16_t h) {
    uint32_t b = (uint32_t)h << 16;
    float f;
    memcpy(&f, &b, 4);
    return f;
}

void orc_gen_bf16(uint64_t seed, uint64_t tid, uint64_t first, uint64_t n, double sigma, uint16_t* out) {
    uint64_t key = orc_splitmix_at(seed, tid);
#pragma omp parallel for schedule(static)
    for (long long i = 0; i < (long long)n; ++i) out[i] = orc_f32_to_bf16(gen_one(key, first + (uint64_t)i, sigma));
}

/* 4-bit block format (see dllm_oracle.h): weight = bf16(d * (q - 8)). */
uint16_t orc_q4_dequant(int code, uint16_t scale_bits) {
    float d = orc_bf16_to_f32(scale_bits);
    float w = d * (float)(code - 8); /* exact: an 8-bit significand times a 4-bit integer */
    return orc_f32_to_bf16(w);
}

int orc_q4_code(uint64_t seed, uint64_t tid, int cols, int r, int c) {
    uint64_t key = orc_splitmix_at(seed, ORC_Q4_CODES + tid);
    return (int)(orc_splitmix_at(key, (uint64_t)r * (uint64_t)cols + (uint64_t)c) >> 60);
}

uint16_t orc_q4_scale(uint64_t seed, uint64_t tid, int cols, int r, int b) {
    uint64_t key = orc_splitmix_at(seed, ORC_Q4_SCALES + tid);
    uint64_t nblk = (uint64_t)(cols + 31) / 32;
    return (uint16_t)(0x3B80u | (uint32_t)(orc_splitmix_at(key, (uint64_t)r * nblk + (uint64_t)b) >> 59));
}

void orc_gen_q4(uint64_t seed, uint64_t tid, int rows, int cols, uint16_t* out) {
#pragma omp parallel for schedule(static)
    for (int r = 0; r < rows; ++r)
        for (int c = 0; c < cols; ++c)
            out[(size_t)r * cols + c] =
                orc_q4_dequant(orc_q4_code(seed, tid, cols, r, c), orc_q4_scale(seed, tid, cols, r, c / 32));
}

/* ------------------------------------------------------------------ */
/* Model                                                                */
/* ------------------------------------------------------------------ */
struct orc_model {
    orc_config c;
    int n_gen_layers;
    uint16_t* embed; /* [V][d], NULL => rows generated on demand */
    uint16_t* head;  /* [V][d] */
    uint16_t** w;    /* per layer: 7 tensors */
    float* norm_attn; /* [L][d] */
    float* norm_ffn;  /* [L][d] */
    float* norm_final; /* [d] */
};

/* Width of the K and V projections: K/V heads x head_dim (grouped-query attention has fewer
 * K/V heads than query heads; n_kv_heads = 0 means as many as query heads). */
static int kv_width(const orc_config* c) {
    return (c->n_kv_heads > 0 ? c->n_kv_heads : c->n_heads) * c->head_dim;
}

static size_t wsize(const orc_config* c, int which, int* rows, int* cols) {
    int d = c->d_model, qd = c->n_heads * c->head_dim, F = c->ffn;
    int r = 0, k = 0;
    switch (which) {
        case ORC_W_Q: r = qd; k = d; break;
        case ORC_W_K: case ORC_W_V: r = kv_width(c); k = d; break;
        case ORC_W_O: r = d; k = qd; break;
        case ORC_W_GATE: case ORC_W_UP: r = F; k = d; break;
        case ORC_W_DOWN: r = d; k = F; break;
    }
    if (rows) *rows = r;
    if (cols) *cols = k;
    return (size_t)r * (size_t)k;
}

static orc_model* model_alloc(const orc_config* c, int n_layers) {
    orc_model* m = (orc_model*)calloc(1, sizeof(orc_model));
    m->c = *c;
    m->n_gen_layers = n_layers;
    m->w = (uint16_t**)calloc((size_t)c->n_layers * 7, sizeof(uint16_t*));
    m->norm_attn = (float*)malloc(sizeof(float) * (size_t)c->n_layers * c->d_model);
    m->norm_ffn = (float*)malloc(sizeof(float) * (size_t)c->n_layers * c->d_model);
    m->norm_final = (float*)malloc(sizeof(float) * (size_t)c->d_model);
    /* RMSNorm gains start at one (their standard initialisation). */
    for (size_t i = 0; i < (size_t)c->n_layers * c->d_model; ++i) m->norm_attn[i] = m->norm_ffn[i] = 1.0f;
    for (int i = 0; i < c->d_model; ++i) m->norm_final[i] = 1.0f;
    return m;
}

orc_model* orc_model_new(const orc_config* c, int gen_layers, int gen_head) {
    int L = gen_layers < 0 || gen_layers > c->n_layers ? c->n_layers : gen_layers;
    orc_model* m = model_alloc(c, L);
    size_t Vd = (size_t)c->vocab * c->d_model;
    if (gen_layers < 0) { /* full model: keep the embedding resident */
        m->embed = (uint16_t*)malloc(Vd * 2);
        orc_gen_bf16(c->weight_seed, ORC_T_EMBED, 0, Vd, 0.02, m->embed);
    }
    const int q4 = c->weight_bits == 4; /* the projections in the 4-bit block format */
    if (gen_head) {
        m->head = (uint16_t*)malloc(Vd * 2);
        if (q4)
            orc_gen_q4(c->weight_seed, ORC_T_HEAD, c->vocab, c->d_model, m->head);
        else
            orc_gen_bf16(c->weight_seed, ORC_T_HEAD, 0, Vd, 0.02, m->head);
    }
    for (int l = 0; l < L; ++l)
        for (int w = 0; w < 7; ++w) {
            int rows = 0, cols = 0;
            size_t n = wsize(c, w, &rows, &cols);
            m->w[l * 7 + w] = (uint16_t*)malloc(n * 2);
            if (q4)
                orc_gen_q4(c->weight_seed, ORC_LAYER_TENSOR(l, w), rows, cols, m->w[l * 7 + w]);
            else
                orc_gen_bf16(c->weight_seed, ORC_LAYER_TENSOR(l, w), 0, n, 0.02, m->w[l * 7 + w]);
        }
    return m;
}

orc_model* orc_model_new_zero(const orc_config* c) {
    orc_model* m = model_alloc(c, c->n_layers);
    size_t Vd = (size_t)c->vocab * c->d_model;
    m->embed = (uint16_t*)calloc(Vd, 2);
    m->head = (uint16_t*)calloc(Vd, 2);
    for (int l = 0; l < c->n_layers; ++l)
        for (int w = 0; w < 7; ++w) m->w[l * 7 + w] = (uint16_t*)calloc(wsize(c, w, NULL, NULL), 2);
    return m;
}

uint16_t* orc_model_weight(orc_model* m, int layer, int which, size_t* n) {
    if (layer < 0) {
        if (n) *n = (size_t)m->c.vocab * m->c.d_model;
        return which == ORC_T_EMBED ? m->embed : (which == ORC_T_HEAD ? m->head : NULL);
    }
    if (layer >= m->n_gen_layers || which < 0 || which > 6) return NULL;
    if (n) *n = wsize(&m->c, which, NULL, NULL);
    return m->w[layer * 7 + which];
}

float* orc_model_norm(orc_model* m, int layer, int which) {
    if (layer < 0) return m->norm_final;
    return (which == 0 ? m->norm_attn : m->norm_ffn) + (size_t)layer * m->c.d_model;
}

void orc_model_free(orc_model* m) {
    if (!m) return;
    for (int i = 0; i < m->c.n_layers * 7; ++i) free(m->w[i]);
    free(m->w);
    free(m->embed);
    free(m->head);
    free(m->norm_attn);
    free(m->norm_ffn);
    free(m->norm_final);
    free(m);
}

/* ------------------------------------------------------------------ */
/* Ops                                                                   */
/* ------------------------------------------------------------------ */

/* RMSNorm: out = x / sqrt(mean(x^2) + eps) * gamma. */
void orc_rmsnorm(int n, const float* x, const float* gamma, double eps, float* out) {
    double ss = 0.0;
    for (int i = 0; i < n; ++i) ss += (double)x[i] * (double)x[i];
    double r = 1.0 / sqrt(ss / n + eps);
    for (int i = 0; i < n; ++i) out[i] = (float)((double)x[i] * r * (double)gamma[i]);
}

/* Rotate-half RoPE at absolute position pos: pairs (i, i + hd/2) rotated by
 * pos * base^(-2i/hd). */
void orc_rope(int hd, double base, int pos, float* v) {
    int h2 = hd / 2;
    for (int i = 0; i < h2; ++i) {
        double theta = pow(base, -2.0 * (double)i / (double)hd);
        double a = (double)pos * theta;
        double c = cos(a), s = sin(a);
        double x1 = v[i], x2 = v[i + h2];
        v[i] = (float)(x1 * c - x2 * s);
        v[i + h2] = (float)(x2 * c + x1 * s);
    }
}

/* y[t][o] = sum_k W[o][k] * x[t][k]  (W bf16 [rows][cols]). */
static void linear(const uint16_t* W, int rows, int cols, const float* x, int T, float* y) {
#pragma omp parallel
    {
        float* wrow = (float*)malloc(sizeof(float) * (size_t)cols);
#pragma omp for schedule(static)
        for (int o = 0; o < rows; ++o) {
            const uint16_t* wr = W + (size_t)o * cols;
            for (int k = 0; k < cols; ++k) wrow[k] = orc_bf16_to_f32(wr[k]);
            for (int t = 0; t < T; ++t) {
                const float* xt = x + (size_t)t * cols;
                double acc = 0.0;
                for (int k = 0; k < cols; ++k) acc += (double)wrow[k] * (double)xt[k];
                y[(size_t)t * rows + o] = (float)acc;
            }
        }
        free(wrow);
    }
}

void orc_decide(int V, int mask_id, const float* z, int32_t cur, int32_t* x0, float* conf, float* tokconf,
                float* margin) {
    int best = -1;
    for (int v = 0; v < V; ++v) {
        if (v == mask_id) continue;
        if (best < 0 || z[v] > z[best]) best = v; /* ties: lowest id */
    }
    double M = z[best];
    double S = 0.0;
    float second = -INFINITY;
    for (int v = 0; v < V; ++v) {
        if (v == mask_id) continue;
        S += exp((double)z[v] - M);
        if (v != best && z[v] > second) second = z[v];
    }
    *x0 = best;
    *conf = (float)(1.0 / S);
    if (cur >= 0 && cur < V && cur != mask_id)
        *tokconf = (float)(exp((double)z[cur] - M) / S);
    else
        *tokconf = 0.0f;
    if (margin) *margin = (float)(M - (double)second);
}

static void embed_row(const orc_model* m, int32_t tok, float* out) {
    int d = m->c.d_model;
    if (m->embed) {
        const uint16_t* e = m->embed + (size_t)tok * d;
        for (int i = 0; i < d; ++i) out[i] = orc_bf16_to_f32(e[i]);
    } else {
        uint16_t* tmp = (uint16_t*)malloc(2 * (size_t)d);
        uint64_t key = orc_splitmix_at(m->c.weight_seed, ORC_T_EMBED);
        for (int i = 0; i < d; ++i) tmp[i] = orc_f32_to_bf16(gen_one(key, (uint64_t)tok * d + i, 0.02));
        for (int i = 0; i < d; ++i) out[i] = orc_bf16_to_f32(tmp[i]);
        free(tmp);
    }
}

int orc_forward(const orc_model* m, int T, const int32_t* tok, const int32_t* pos, int P, const float* pk,
                const float* pv, const int32_t* group, float* out_k, float* out_v, float* logits,
                int n_layers_run) {
    return orc_forward_ex(m, T, T, tok, pos, P, pk, pv, group, out_k, out_v, logits, n_layers_run);
}

int orc_forward_ex(const orc_model* m, int T, int Tk, const int32_t* tok, const int32_t* pos, int P, const float* pk,
                   const float* pv, const int32_t* group, float* out_k, float* out_v, float* logits,
                   int n_layers_run) {
    const orc_config* c = &m->c;
    int d = c->d_model, H = c->n_heads, hd = c->head_dim, F = c->ffn, V = c->vocab;
    int qd = H * hd;
    /* grouped-query attention: query head hh reads K/V head hh / grp */
    int kvd = kv_width(c), Hkv = kvd / hd, grp = H / Hkv;
    if (Hkv < 1 || H % Hkv) return -1;
    int L = n_layers_run < 0 || n_layers_run > c->n_layers ? c->n_layers : n_layers_run;
    if (L > m->n_gen_layers) return -1;
    if (T <= 0) return 0;
    if (Tk < 0 || Tk > T) return -1;
    size_t Td = (size_t)T * d;
    float* x = (float*)malloc(sizeof(float) * Td);
    float* h = (float*)malloc(sizeof(float) * Td);
    float* q = (float*)malloc(sizeof(float) * (size_t)T * qd);
    float* k = (float*)malloc(sizeof(float) * (size_t)T * kvd);
    float* v = (float*)malloc(sizeof(float) * (size_t)T * kvd);
    float* att = (float*)malloc(sizeof(float) * (size_t)T * qd);
    float* o = (float*)malloc(sizeof(float) * Td);
    float* g = (float*)malloc(sizeof(float) * (size_t)T * F);
    float* u = (float*)malloc(sizeof(float) * (size_t)T * F);
    double scale = 1.0 / sqrt((double)hd);

    for (int t = 0; t < T; ++t) embed_row(m, tok[t], x + (size_t)t * d);

    for (int l = 0; l < L; ++l) {
        uint16_t* const* W = m->w + (size_t)l * 7;
        /* attention sub-layer */
        for (int t = 0; t < T; ++t)
            orc_rmsnorm(d, x + (size_t)t * d, m->norm_attn + (size_t)l * d, c->rms_eps, h + (size_t)t * d);
        linear(W[ORC_W_Q], qd, d, h, T, q);
        linear(W[ORC_W_K], kvd, d, h, T, k);
        linear(W[ORC_W_V], kvd, d, h, T, v);
        for (int t = 0; t < T; ++t) {
            for (int hh = 0; hh < H; ++hh) orc_rope(hd, c->rope_base, pos[t], q + (size_t)t * qd + (size_t)hh * hd);
            for (int hh = 0; hh < Hkv; ++hh) orc_rope(hd, c->rope_base, pos[t], k + (size_t)t * kvd + (size_t)hh * hd);
        }
        if (out_k) memcpy(out_k + (size_t)l * T * kvd, k, sizeof(float) * (size_t)T * kvd);
        if (out_v) memcpy(out_v + (size_t)l * T * kvd, v, sizeof(float) * (size_t)T * kvd);
        const float* lk = P > 0 ? pk + (size_t)l * P * kvd : NULL;
        const float* lv = P > 0 ? pv + (size_t)l * P * kvd : NULL;
        int NK = P + Tk; /* rows from Tk on are queries only */
#pragma omp parallel
        {
            double* sc = (double*)malloc(sizeof(double) * (size_t)NK);
            double* acc = (double*)malloc(sizeof(double) * (size_t)hd);
#pragma omp for collapse(2) schedule(static)
            for (int hh = 0; hh < H; ++hh)
                for (int t = 0; t < T; ++t) {
                    const float* qt = q + (size_t)t * qd + (size_t)hh * hd;
                    const size_t kh = (size_t)(hh / grp) * hd; /* its K/V head */
                    double mx = -INFINITY;
                    /* keys in position order: cached prefix, then the window */
                    for (int j = 0; j < NK; ++j) {
                        const float* kj;
                        if (j < P) {
                            kj = lk + (size_t)j * kvd + kh;
                        } else {
                            int w = j - P;
                            if (group && group[w] > group[t]) { sc[j] = -INFINITY; continue; }
                            kj = k + (size_t)w * kvd + kh;
                        }
                        double s = 0.0;
                        for (int i = 0; i < hd; ++i) s += (double)qt[i] * (double)kj[i];
                        sc[j] = s * scale;
                        if (sc[j] > mx) mx = sc[j];
                    }
                    double sum = 0.0;
                    for (int j = 0; j < NK; ++j) {
                        sc[j] = sc[j] == -INFINITY ? 0.0 : exp(sc[j] - mx);
                        sum += sc[j];
                    }
                    for (int i = 0; i < hd; ++i) acc[i] = 0.0;
                    for (int j = 0; j < NK; ++j) {
                        if (sc[j] == 0.0) continue;
                        const float* vj = j < P ? lv + (size_t)j * kvd + kh : v + (size_t)(j - P) * kvd + kh;
                        double p = sc[j] / sum;
                        for (int i = 0; i < hd; ++i) acc[i] += p * (double)vj[i];
                    }
                    float* ot = att + (size_t)t * qd + (size_t)hh * hd;
                    for (int i = 0; i < hd; ++i) ot[i] = (float)acc[i];
                }
            free(sc);
            free(acc);
        }
        linear(W[ORC_W_O], d, qd, att, T, o);
        for (size_t i = 0; i < Td; ++i) x[i] += o[i];
        /* MLP sub-layer (SwiGLU) */
        for (int t = 0; t < T; ++t)
            orc_rmsnorm(d, x + (size_t)t * d, m->norm_ffn + (size_t)l * d, c->rms_eps, h + (size_t)t * d);
        linear(W[ORC_W_GATE], F, d, h, T, g);
        linear(W[ORC_W_UP], F, d, h, T, u);
        for (size_t i = 0; i < (size_t)T * F; ++i) {
            double gg = g[i];
            g[i] = (float)(gg / (1.0 + exp(-gg)) * (double)u[i]);
        }
        linear(W[ORC_W_DOWN], d, F, g, T, o);
        for (size_t i = 0; i < Td; ++i) x[i] += o[i];
    }
    if (logits) {
        if (!m->head) return -2;
        for (int t = 0; t < T; ++t) orc_rmsnorm(d, x + (size_t)t * d, m->norm_final, c->rms_eps, h + (size_t)t * d);
        linear(m->head, V, d, h, T, logits);
    }
    free(x); free(h); free(q); free(k); free(v); free(att); free(o); free(g); free(u);
    return 0;
}

/* ------------------------------------------------------------------ */
/* Commit / re-mask / drafts                                             */
/* ------------------------------------------------------------------ */
/* Order of one pass (all on the same step's decisions):
 *   1. revision (Sec. 3.3): committed-but-unstable tokens of the current
 *      block reaching theta_stable become STABLE; those below theta_remask
 *      are re-masked, at most remask_max per step, lowest confidence first.
 *      Enabled when theta_remask > 0, skipped on the block's last step.
 *   2. schedule: k = ceil(m / (S - step)) commits, m = masked count.
 *   3. commit (Sec. 2.1): the k masked positions of the current block with
 *      the highest confidence (ties: lower position) take their argmax.
 *   4. drafts (Sec. 3.2): with the prefix cache on and lookahead active,
 *      each future block in the window drafts its most confident masked
 *      position. */
int orc_commit(const orc_sched* s, int mask_id, int n_pos, int32_t* tok, uint8_t* st, int w0, int T, int c0,
               int c1, int step, const int32_t* x0, const float* conf, const float* tokconf, orc_step_out* out) {
    orc_step_out r;
    memset(&r, 0, sizeof(r));
    int S = s->steps_per_block;
    if (c1 > w0 + T || c1 > n_pos || c0 > c1 || w0 > c1) return -1;
    /* block positions left of the window (continuous sliding) are settled */
    for (int p = c0; p < w0 && p < c1; ++p)
        if (st[p] == ORC_MASKED || st[p] == ORC_DRAFT) return -1;
    if (s->theta_remask > 0.0f && step < S - 1) {
        int r0 = c0 > w0 ? c0 : w0; /* the revision reaches only the block positions in the window */
        for (int p = r0; p < c1; ++p)
            if (st[p] == ORC_COMMITTED && tokconf[p - w0] >= s->theta_stable) {
                st[p] = ORC_STABLE;
                r.n_stable++;
            }
        /* candidates ranked by (tokconf ascending, position ascending) */
        int* sel = (int*)malloc(sizeof(int) * (size_t)(c1 - c0 + 1));
        int nsel = 0;
        for (int p = r0; p < c1; ++p) {
            if (st[p] != ORC_COMMITTED || !(tokconf[p - w0] < s->theta_remask)) continue;
            int rank = 0;
            for (int q = r0; q < c1; ++q) {
                if (q == p || st[q] != ORC_COMMITTED || !(tokconf[q - w0] < s->theta_remask)) continue;
                float a = tokconf[q - w0], b = tokconf[p - w0];
                if (a < b || (a == b && q < p)) rank++;
            }
            if (rank < s->remask_max) sel[nsel++] = p;
        }
        for (int i = 0; i < nsel; ++i) {
            st[sel[i]] = ORC_MASKED;
            tok[sel[i]] = mask_id;
        }
        r.n_remasked = nsel;
        free(sel);
    }
    int m = 0;
    for (int p = c0; p < c1; ++p) m += st[p] == ORC_MASKED;
    int nc = 0;
    if (s->commit_mode == ORC_COMMIT_THRESHOLD) {
        /* Sec. 3.3: masked positions at or above theta_visible take their prediction and become
         * visible, or stable when they also reach theta_stable */
        for (int p = c0; p < c1; ++p) {
            if (st[p] != ORC_MASKED || !(conf[p - w0] >= s->theta_visible)) continue;
            tok[p] = x0[p - w0];
            if (conf[p - w0] >= s->theta_stable) {
                st[p] = ORC_STABLE;
                r.n_stable++;
            } else {
                st[p] = ORC_COMMITTED;
            }
            nc++;
        }
        /* none did: the most confident masked position (the first of equals) becomes visible */
        if (nc == 0 && m > 0) {
            int best = -1;
            for (int p = c0; p < c1; ++p)
                if (st[p] == ORC_MASKED && (best < 0 || conf[p - w0] > conf[best - w0])) best = p;
            tok[best] = x0[best - w0];
            st[best] = ORC_COMMITTED;
            nc = 1;
        }
    } else {
        int left = S - step;
        int k = m == 0 ? 0 : (left <= 1 ? m : (m + left - 1) / left);
        int* committed = (int*)malloc(sizeof(int) * (size_t)(c1 - c0 + 1));
        for (int p = c0; p < c1; ++p) {
            if (st[p] != ORC_MASKED) continue;
            int rank = 0;
            for (int q = c0; q < c1; ++q) {
                if (q == p || st[q] != ORC_MASKED) continue;
                float a = conf[q - w0], b = conf[p - w0];
                if (a > b || (a == b && q < p)) rank++;
            }
            if (rank < k) committed[nc++] = p;
        }
        for (int i = 0; i < nc; ++i) {
            int p = committed[i];
            tok[p] = x0[p - w0];
            st[p] = ORC_COMMITTED;
        }
        free(committed);
    }
    r.n_committed = nc;
    if (s->use_prefix_cache && (s->spec_blocks > 0 || s->slide)) { /* future blocks in the window */
        int w1 = w0 + T;
        for (int b0 = c1; b0 < w1; b0 += s->block_len) {
            int b1 = b0 + s->block_len < w1 ? b0 + s->block_len : w1;
            int best = -1;
            for (int p = b0; p < b1; ++p) {
                if (st[p] != ORC_MASKED) continue;
                if (best < 0 || conf[p - w0] > conf[best - w0]) best = p;
            }
            if (best >= 0) {
                tok[best] = x0[best - w0];
                st[best] = ORC_DRAFT;
                r.n_drafts++;
            }
        }
    }
    r.masked_after = m - nc;
    r.block_done = r.masked_after == 0;
    if (out) *out = r;
    return 0;
}

/* ------------------------------------------------------------------ */
/* Session                                                               */
/* ------------------------------------------------------------------ */
struct orc_session {
    const orc_model* m;
    orc_sched s;
    int Lp, G, n_pos;
    int32_t* tok;
    uint8_t* st;
    float* pk; /* [L][n_pos][kvd]: K/V heads x head_dim */
    float* pv;
    int kv_len;
    int cb, c0, c1, step; /* current block */
    /* last step */
    int w0, T, spec_on;
    int32_t* x0;
    float *conf, *tokconf, *margin, *logits;
    /* sparse cache refresh of the last step: tracked positions and their decisions */
    int scr_n;
    int32_t *scr_pos, *scr_x0;
    float *scr_conf, *scr_tokconf, *scr_margin;
};

orc_session* orc_session_new(const orc_model* m, const orc_sched* s, int Lp, const int32_t* prompt, int G) {
    orc_session* x = (orc_session*)calloc(1, sizeof(orc_session));
    const orc_config* c = &m->c;
    x->m = m;
    x->s = *s;
    x->Lp = Lp;
    x->G = G;
    x->n_pos = Lp + G;
    x->tok = (int32_t*)malloc(sizeof(int32_t) * (size_t)x->n_pos);
    x->st = (uint8_t*)malloc((size_t)x->n_pos);
    for (int i = 0; i < Lp; ++i) { x->tok[i] = prompt[i]; x->st[i] = ORC_FIXED; }
    for (int i = Lp; i < x->n_pos; ++i) { x->tok[i] = c->mask_id; x->st[i] = ORC_MASKED; }
    size_t kvn = (size_t)c->n_layers * x->n_pos * kv_width(c);
    x->pk = (float*)calloc(kvn, sizeof(float));
    x->pv = (float*)calloc(kvn, sizeof(float));
    x->cb = -1;
    x->x0 = (int32_t*)calloc((size_t)x->n_pos, sizeof(int32_t));
    x->conf = (float*)calloc((size_t)x->n_pos, sizeof(float));
    x->tokconf = (float*)calloc((size_t)x->n_pos, sizeof(float));
    x->margin = (float*)calloc((size_t)x->n_pos, sizeof(float));
    return x;
}

void orc_session_free(orc_session* x) {
    if (!x) return;
    free(x->tok); free(x->st); free(x->pk); free(x->pv);
    free(x->x0); free(x->conf); free(x->tokconf); free(x->margin); free(x->logits);
    free(x->scr_pos); free(x->scr_x0); free(x->scr_conf); free(x->scr_tokconf); free(x->scr_margin);
    free(x);
}

int orc_scr_decisions(const orc_session* x, int32_t* pos, int32_t* x0, float* conf, float* tokconf, float* margin) {
    int n = x->scr_n;
    if (n <= 0) return 0;
    if (pos) memcpy(pos, x->scr_pos, sizeof(int32_t) * (size_t)n);
    if (x0) memcpy(x0, x->scr_x0, sizeof(int32_t) * (size_t)n);
    if (conf) memcpy(conf, x->scr_conf, sizeof(float) * (size_t)n);
    if (tokconf) memcpy(tokconf, x->scr_tokconf, sizeof(float) * (size_t)n);
    if (margin) memcpy(margin, x->scr_margin, sizeof(float) * (size_t)n);
    return n;
}

int orc_n_pos(const orc_session* x) { return x->n_pos; }

/* Run the layers over positions [a, b) with P = kv_len cached keys and
 * append their K/V to the prefix cache (prompt prefill and finished-block
 * append use the same rule: attend to prefix plus the new positions). */
static int append_kv(orc_session* x, int a, int b) {
    const orc_config* c = &x->m->c;
    int T = b - a, kvd = kv_width(c), L = c->n_layers;
    if (T <= 0) return 0;
    int P = x->kv_len;
    int32_t* pos = (int32_t*)malloc(sizeof(int32_t) * (size_t)T);
    for (int t = 0; t < T; ++t) pos[t] = a + t;
    float* pk = NULL;
    float* pv = NULL;
    if (P > 0) { /* contiguous [L][P][kvd] view of the cache */
        pk = (float*)malloc(sizeof(float) * (size_t)L * P * kvd);
        pv = (float*)malloc(sizeof(float) * (size_t)L * P * kvd);
        for (int l = 0; l < L; ++l) {
            memcpy(pk + (size_t)l * P * kvd, x->pk + (size_t)l * x->n_pos * kvd, sizeof(float) * (size_t)P * kvd);
            memcpy(pv + (size_t)l * P * kvd, x->pv + (size_t)l * x->n_pos * kvd, sizeof(float) * (size_t)P * kvd);
        }
    }
    float* ok = (float*)malloc(sizeof(float) * (size_t)L * T * kvd);
    float* ov = (float*)malloc(sizeof(float) * (size_t)L * T * kvd);
    int rc = orc_forward(x->m, T, x->tok + a, pos, P, pk, pv, NULL, ok, ov, NULL, -1);
    for (int l = 0; l < L; ++l) {
        memcpy(x->pk + ((size_t)l * x->n_pos + P) * kvd, ok + (size_t)l * T * kvd, sizeof(float) * (size_t)T * kvd);
        memcpy(x->pv + ((size_t)l * x->n_pos + P) * kvd, ov + (size_t)l * T * kvd, sizeof(float) * (size_t)T * kvd);
    }
    x->kv_len = P + T;
    free(pos); free(pk); free(pv); free(ok); free(ov);
    return rc;
}

int orc_prefill(orc_session* x) {
    x->kv_len = 0;
    if (!x->s.use_prefix_cache) return 0;
    return append_kv(x, 0, x->Lp);
}

int orc_begin_block(orc_session* x) {
    int bl = x->s.block_len;
    if (x->cb >= 0) {
        for (int p = x->c0; p < x->c1; ++p)
            if (x->st[p] == ORC_MASKED) return -3; /* block not finished */
        if (x->s.use_prefix_cache) {
            int rc = append_kv(x, x->kv_len, x->c1); /* what has not slid into the cache yet */
            if (rc) return rc;
        }
    }
    int nb = x->cb + 1;
    int c0 = x->Lp + nb * bl;
    if (c0 >= x->n_pos) { x->cb = nb; x->c0 = x->c1 = x->n_pos; return 1; }
    x->cb = nb;
    x->c0 = c0;
    x->c1 = c0 + bl < x->n_pos ? c0 + bl : x->n_pos;
    x->step = 0;
    /* drafts of the new current block are accepted provisionally; the
     * revision pass re-checks them (Sec. 3.2) */
    for (int p = x->c0; p < x->c1; ++p)
        if (x->st[p] == ORC_DRAFT) x->st[p] = ORC_COMMITTED;
    return 0;
}

int orc_denoise_step(orc_session* x, orc_step_out* out, int keep_logits) {
    const orc_config* c = &x->m->c;
    int V = c->vocab, kvd = kv_width(c), L = c->n_layers;
    if (x->cb < 0 || x->c0 >= x->n_pos) return -3;
    int masked = 0;
    for (int p = x->c0; p < x->c1; ++p) masked += x->st[p] == ORC_MASKED;
    int w0, w1, spec = 0;
    if (x->s.use_prefix_cache) {
        w0 = x->kv_len;
        /* the window without lookahead: the current block, or with sliding one block's length
         * from the frontier */
        int base = x->s.slide ? w0 + x->s.block_len : x->c1;
        if (base > x->n_pos) base = x->n_pos;
        w1 = base;
        if (x->s.spec_blocks > 0 && masked <= x->s.spec_trigger && base < x->n_pos) {
            int k = x->s.spec_blocks;
            if (x->s.spec_allowance >= 0.0f && x->s.spec_lat_n > 0) {
                /* greedy: one more future block while the step stays within the allowance */
                int i0 = (base - w0 + x->s.block_len - 1) / x->s.block_len - 1;
                k = 0;
                for (int j = 1; j <= x->s.spec_blocks; ++j) {
                    int i = i0 + j;
                    if (i0 < 0 || i >= x->s.spec_lat_n || i0 >= x->s.spec_lat_n) break;
                    if (x->s.spec_lat[i] > (1.0f + x->s.spec_allowance) * x->s.spec_lat[i0]) break;
                    k = j;
                }
            }
            if (k > 0) {
                spec = 1;
                w1 = base + k * x->s.block_len;
                if (w1 > x->n_pos) w1 = x->n_pos;
            }
        }
    } else {
        w0 = 0;
        w1 = x->n_pos;
    }
    int T = w1 - w0, P = x->s.use_prefix_cache ? x->kv_len : 0;
    x->w0 = w0; x->T = T; x->spec_on = spec;
    /* sparse cache refresh: the first scr_rows visible (COMMITTED) prefix positions ride along
     * as query-only rows */
    int R = x->s.use_prefix_cache ? x->s.scr_rows : 0, nt = 0;
    if (R > 0 && !x->scr_pos) {
        x->scr_pos = (int32_t*)calloc((size_t)R, sizeof(int32_t));
        x->scr_x0 = (int32_t*)calloc((size_t)R, sizeof(int32_t));
        x->scr_conf = (float*)calloc((size_t)R, sizeof(float));
        x->scr_tokconf = (float*)calloc((size_t)R, sizeof(float));
        x->scr_margin = (float*)calloc((size_t)R, sizeof(float));
    }
    for (int p = 0; p < x->kv_len && nt < R; ++p)
        if (x->st[p] == ORC_COMMITTED) x->scr_pos[nt++] = p;
    x->scr_n = nt;
    int Tq = T + nt;
    int32_t* pos = (int32_t*)malloc(sizeof(int32_t) * (size_t)Tq);
    int32_t* rows = (int32_t*)malloc(sizeof(int32_t) * (size_t)Tq);
    for (int t = 0; t < T; ++t) { pos[t] = w0 + t; rows[t] = x->tok[w0 + t]; }
    for (int r = 0; r < nt; ++r) { pos[T + r] = x->scr_pos[r]; rows[T + r] = x->tok[x->scr_pos[r]]; }
    float* pk = NULL;
    float* pv = NULL;
    if (P > 0) {
        pk = (float*)malloc(sizeof(float) * (size_t)L * P * kvd);
        pv = (float*)malloc(sizeof(float) * (size_t)L * P * kvd);
        for (int l = 0; l < L; ++l) {
            memcpy(pk + (size_t)l * P * kvd, x->pk + (size_t)l * x->n_pos * kvd, sizeof(float) * (size_t)P * kvd);
            memcpy(pv + (size_t)l * P * kvd, x->pv + (size_t)l * x->n_pos * kvd, sizeof(float) * (size_t)P * kvd);
        }
    }
    free(x->logits);
    x->logits = (float*)malloc(sizeof(float) * (size_t)Tq * V);
    int keep_kv = nt > 0 || x->s.slide;
    float* nk = keep_kv ? (float*)malloc(sizeof(float) * (size_t)L * Tq * kvd) : NULL;
    float* nv = keep_kv ? (float*)malloc(sizeof(float) * (size_t)L * Tq * kvd) : NULL;
    int rc = orc_forward_ex(x->m, Tq, T, rows, pos, P, pk, pv, NULL, nk, nv, x->logits, -1);
    free(pos); free(rows); free(pk); free(pv);
    if (rc) { free(nk); free(nv); return rc; }
    for (int t = 0; t < T; ++t)
        orc_decide(V, c->mask_id, x->logits + (size_t)t * V, x->tok[w0 + t], x->x0 + t, x->conf + t, x->tokconf + t,
                   x->margin + t);
    for (int r = 0; r < nt; ++r)
        orc_decide(V, c->mask_id, x->logits + (size_t)(T + r) * V, x->tok[x->scr_pos[r]], x->scr_x0 + r,
                   x->scr_conf + r, x->scr_tokconf + r, x->scr_margin + r);
    if (!keep_logits) { free(x->logits); x->logits = NULL; }
    /* continuous sliding: the block positions visible when the forward ran */
    int nb_win = x->c1 - w0 > 0 ? x->c1 - w0 : 0;
    uint8_t* vis0 = (uint8_t*)malloc((size_t)nb_win + 1);
    for (int t = 0; t < nb_win; ++t) vis0[t] = x->st[w0 + t] == ORC_COMMITTED || x->st[w0 + t] == ORC_STABLE;
    orc_step_out so;
    rc = orc_commit(&x->s, c->mask_id, x->n_pos, x->tok, x->st, w0, T, x->c0, x->c1, x->step, x->x0, x->conf,
                    x->tokconf, &so);
    /* the tracked positions: re-scored, then their refreshed K/V merged at the step boundary */
    for (int r = 0; r < nt && !rc; ++r) {
        int p = x->scr_pos[r];
        float tc = x->scr_tokconf[r];
        if (tc >= x->s.theta_stable) {
            x->st[p] = ORC_STABLE;
            so.n_stable++;
        } else if (x->s.theta_remask > 0.0f && tc < x->s.theta_remask && x->scr_x0[r] != x->tok[p]) {
            x->tok[p] = x->scr_x0[r];
            so.n_revised++;
            continue;
        }
        for (int l = 0; l < L; ++l) {
            memcpy(x->pk + ((size_t)l * x->n_pos + p) * kvd, nk + ((size_t)l * Tq + T + r) * kvd, sizeof(float) * kvd);
            memcpy(x->pv + ((size_t)l * x->n_pos + p) * kvd, nv + ((size_t)l * Tq + T + r) * kvd, sizeof(float) * kvd);
        }
        so.n_refreshed++;
    }
    /* continuous sliding: the leading run of positions visible before and after the commit pass
     * takes the K/V this forward computed (from those same ids) into the cache */
    if (x->s.slide && !rc) {
        int adv = 0;
        while (adv < nb_win && vis0[adv] &&
               (x->st[w0 + adv] == ORC_COMMITTED || x->st[w0 + adv] == ORC_STABLE))
            adv++;
        for (int l = 0; l < L; ++l)
            for (int t = 0; t < adv; ++t) {
                memcpy(x->pk + ((size_t)l * x->n_pos + w0 + t) * kvd, nk + ((size_t)l * Tq + t) * kvd, sizeof(float) * kvd);
                memcpy(x->pv + ((size_t)l * x->n_pos + w0 + t) * kvd, nv + ((size_t)l * Tq + t) * kvd, sizeof(float) * kvd);
            }
        x->kv_len += adv;
    }
    free(vis0);
    free(nk); free(nv);
    if (out) *out = so;
    x->step++;
    return rc;
}

int orc_window(const orc_session* x, int32_t* info) {
    info[0] = x->w0; info[1] = x->T; info[2] = x->c0; info[3] = x->c1;
    info[4] = x->step; info[5] = x->kv_len; info[6] = x->spec_on;
    return 0;
}

int orc_step_decisions(const orc_session* x, int32_t* x0, float* conf, float* tokconf, float* margin, float* logits) {
    int T = x->T;
    if (x0) memcpy(x0, x->x0, sizeof(int32_t) * (size_t)T);
    if (conf) memcpy(conf, x->conf, sizeof(float) * (size_t)T);
    if (tokconf) memcpy(tokconf, x->tokconf, sizeof(float) * (size_t)T);
    if (margin) memcpy(margin, x->margin, sizeof(float) * (size_t)T);
    if (logits) {
        if (!x->logits) return -4;
        memcpy(logits, x->logits, sizeof(float) * (size_t)T * x->m->c.vocab);
    }
    return 0;
}

int orc_get_state(const orc_session* x, int32_t* tok, uint8_t* st, int32_t* kv_len) {
    if (tok) memcpy(tok, x->tok, sizeof(int32_t) * (size_t)x->n_pos);
    if (st) memcpy(st, x->st, (size_t)x->n_pos);
    if (kv_len) *kv_len = x->kv_len;
    return 0;
}

int orc_set_state(orc_session* x, const int32_t* tok, const uint8_t* st) {
    if (tok) memcpy(x->tok, tok, sizeof(int32_t) * (size_t)x->n_pos);
    if (st) memcpy(x->st, st, (size_t)x->n_pos);
    return 0;
}

const float* orc_prefix_kv(const orc_session* x, int layer, int which) {
    const orc_config* c = &x->m->c;
    size_t off = (size_t)layer * x->n_pos * kv_width(c);
    return (which == 0 ? x->pk : x->pv) + off;
}
