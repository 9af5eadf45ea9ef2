// C ABI of the denoising path (include/dllm.h): device memory layout,
// request state, and the host sequencing of the step's kernels.
//
// HBM layout (one arena, offsets fixed at init):
//   weights  per layer: Wqkv [3*qd (pad 128)][d], Wo [d][qd],
//            Wgu [ceil(F/64)*128][d] (64 gate rows then 64 up rows per
//            128-row tile), Wd [d][F]; embedding [V][d]; LM head [V pad 128][d]
//   KV cache [L][K|V][batch][head][position][head_dim] bf16
//   activations for max_batch * max_window tokens (fp32 residual, bf16 GEMM
//   operands), attention and GEMM split partials, LM-head tile statistics
//   request state: ids int32 [batch][max_ctx], token states uint8, plan.
#include "../../include/dllm.h"
#include "../../include/dllm_ops.h"
#include "internal.h"

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

using namespace dllm;

namespace {

constexpr int kMaxSMs = 256;  // upper bound for scratch sizing

size_t al256(size_t x) { return (x + 255) & ~size_t(255); }
int rup(int x, int m) { return (x + m - 1) / m * m; }

struct Layout {
    int qd, kvd, Hkv, qkv_rows, gu_rows, d_rows, o_rows, head_rows, head_tiles, max_tok;
    size_t off_w, per_layer, off_emb, off_head, off_kv, kv_half;
    size_t off_x, off_xn, off_q, off_attn, off_h, off_sq, off_theta;
    int n_sq;
    size_t off_lmp, off_zcur, off_cur, off_x0, off_conf, off_tokconf;
    size_t off_part, part_floats, off_cnt, off_done, off_epoch, off_trk, off_smerge, off_side;
    size_t off_xc, off_sqc, off_curc, off_rmap, off_nrows;
    int cnt_len, done_len;  // per phase slot
    size_t off_tok, off_st, off_stok, off_sst, off_seqkv, off_plan, off_outs, off_status;
    size_t total;
    size_t w_qkv, w_o, w_gu, w_d;  // element offsets inside a layer (bf16) or byte offsets (4-bit)
    bool q4;                       // projections in the 4-bit block format (kQ4TileBytes tiles)
};

Layout make_layout(const dllm_config& c) {
    Layout L{};
    const int d = c.d_model, H = c.n_heads, hd = c.head_dim, F = c.ffn, V = c.vocab;
    L.qd = H * hd;
    L.Hkv = c.n_kv_heads > 0 ? c.n_kv_heads : H;  // grouped-query attention: fewer K/V heads
    L.kvd = L.Hkv * hd;
    L.qkv_rows = rup(L.qd + 2 * L.kvd, 128);
    L.o_rows = rup(d, 128);
    L.gu_rows = (F + 63) / 64 * 128;
    L.d_rows = rup(d, 128);
    L.head_rows = rup(V, 128);
    L.head_tiles = L.head_rows / 128;
    L.max_tok = c.max_batch * c.max_window;
    L.q4 = c.weight_bits == 4;
    if (L.q4) {  // byte offsets of tile-major 4-bit matrices: (rows / 128) x (K / 64) tiles each
        auto tiles = [](int rows, int k) { return static_cast<size_t>(rows / 128) * ((k + 63) / 64) * kQ4TileBytes; };
        L.w_qkv = 0;
        L.w_o = L.w_qkv + tiles(L.qkv_rows, d);
        L.w_gu = L.w_o + tiles(L.o_rows, L.qd);
        L.w_d = L.w_gu + tiles(L.gu_rows, d);
        L.per_layer = L.w_d + tiles(L.d_rows, F);
    } else {
        L.w_qkv = 0;
        L.w_o = L.w_qkv + static_cast<size_t>(L.qkv_rows) * d;
        L.w_gu = L.w_o + static_cast<size_t>(L.o_rows) * L.qd;
        L.w_d = L.w_gu + static_cast<size_t>(L.gu_rows) * d;
        L.per_layer = L.w_d + static_cast<size_t>(L.d_rows) * rup(F, 64);  // tile-major: K padded to 64
    }
    size_t o = 0;
    auto take = [&](size_t bytes) {
        size_t r = o;
        o = al256(o + bytes);
        return r;
    };
    L.off_w = take(L.per_layer * (L.q4 ? 1 : 2) * c.n_layers);
    L.off_emb = take(static_cast<size_t>(V) * d * 2);
    L.off_head = take(L.q4 ? static_cast<size_t>(L.head_tiles) * ((d + 63) / 64) * kQ4TileBytes
                           : static_cast<size_t>(L.head_rows) * d * 2);
    L.kv_half = static_cast<size_t>(c.max_batch) * L.Hkv * c.max_ctx * hd;
    L.off_kv = take(L.kv_half * 2 * 2 * c.n_layers);
    const size_t T = L.max_tok;
    L.off_x = take(T * d * 4);
    L.off_xn = take(T * std::max(d, L.qd) * 2);
    L.off_q = take(T * L.qd * 2);
    L.off_attn = take(T * L.qd * 2);
    L.off_h = take(T * F * 2);
    L.n_sq = (d + 127) / 128;
    L.off_sq = take(static_cast<size_t>(L.n_sq) * T * 4);
    L.off_theta = take(static_cast<size_t>(hd / 2) * 4);
    L.off_lmp = take(static_cast<size_t>(L.head_tiles) * T * 3 * 4);
    L.off_zcur = take(T * 4);
    L.off_cur = take(T * 4);
    L.off_x0 = take(T * 4);
    L.off_conf = take(T * 4);
    L.off_tokconf = take(T * 4);
    // chained projections: per phase slot, split partials (one per CTA), tile tickets (one per
    // 128-byte line) and tile completion flags
    L.part_floats = static_cast<size_t>(kMaxSMs) * 256 * 128;
    L.off_part = take(L.part_floats * 4 * kMaxPhases);
    const int mt_max = std::max(std::max(L.head_tiles, L.gu_rows / 128), std::max(L.qkv_rows, L.d_rows) / 128);
    L.done_len = mt_max * ((L.max_tok + 255) / 256 + 1);
    L.cnt_len = L.done_len * 32;
    L.off_cnt = take(static_cast<size_t>(L.cnt_len) * 4 * kMaxPhases);
    L.off_done = take(static_cast<size_t>(L.done_len) * 4 * kMaxPhases * 2);  // done, then done2 slots
    L.off_epoch = take(256);
    const size_t S = static_cast<size_t>(c.max_batch) * c.max_ctx;
    L.off_tok = take(S * 4);
    L.off_st = take(S);
    L.off_stok = take(S * 4);
    L.off_sst = take(S);
    L.off_seqkv = take(static_cast<size_t>(c.max_batch) * 4);
    L.off_plan = take(static_cast<size_t>(c.max_batch) * 16);
    L.off_outs = take(static_cast<size_t>(c.max_batch) * 32);
    L.off_status = take(16);
    // sparse cache refresh: tracked positions and merge flags [B][R], side K/V
    // [L][2][B][Hkv][R][hd] (R <= DLLM_MAX_SCR_ROWS)
    L.off_trk = take(static_cast<size_t>(c.max_batch) * DLLM_MAX_SCR_ROWS * 4);
    L.off_smerge = take(static_cast<size_t>(c.max_batch) * DLLM_MAX_SCR_ROWS * 4);
    L.off_side = take(static_cast<size_t>(c.n_layers) * 2 * c.max_batch * L.kvd * DLLM_MAX_SCR_ROWS * 2);
    // selective logits skipping: the compacted LM-head operand (bf16 rows, RMSNorm statistics,
    // current ids), the row map and the row count
    L.off_xc = take(T * d * 2);
    L.off_sqc = take(static_cast<size_t>(L.n_sq) * T * 4);
    L.off_curc = take(T * 4);
    L.off_rmap = take(T * 4);
    L.off_nrows = take(16);
    L.total = o;
    return L;
}

const char* check_cfg(const dllm_config& c) {
    if (c.n_layers < 1 || c.d_model < 64 || c.n_heads < 1 || c.ffn < 8 || c.vocab < 2) return "bad model shape";
    if (c.head_dim != 64 && c.head_dim != 128) return "head_dim must be 64 or 128";
    if (c.d_model % 128 || (c.n_heads * c.head_dim) % 128)
        return "d_model and n_heads*head_dim must be multiples of 128";
    if (c.n_kv_heads < 0 || (c.n_kv_heads > 0 && (c.n_heads % c.n_kv_heads || (c.n_kv_heads * c.head_dim) % 128)))
        return "n_kv_heads must divide n_heads, with n_kv_heads*head_dim a multiple of 128";
    if (c.ffn % 8 || c.vocab % 8) return "ffn and vocab must be multiples of 8";
    if (c.mask_id < 0 || c.mask_id >= c.vocab) return "mask_id out of range";
    if (c.max_batch < 1 || c.max_ctx < 1 || c.max_window < 1 || c.block_len < 1) return "bad capacities";
    if (c.max_batch * c.max_window > 4096) return "max_batch * max_window must be <= 4096";
    if (c.max_batch > 256) return "max_batch must be <= 256";
    if (c.block_len > kMaxBlock) return "block_len too large";
    if (c.rms_eps <= 0.0f || c.rope_base <= 1.0f) return "bad rope_base / rms_eps";
    if (c.weight_bits != 0 && c.weight_bits != 16 && c.weight_bits != 4) return "weight_bits must be 16 or 4";
    return nullptr;
}

}  // namespace

struct dllm_ctx {
    dllm_config cfg{};
    Layout L{};
    int sms = 0;
    cudaStream_t stream = nullptr;
    bool own_stream = false;
    uint8_t* arena = nullptr;
    bool own_arena = false;
    // views
    __nv_bfloat16* emb = nullptr;
    uint8_t* head = nullptr;         // LM head: bf16 or 4-bit tiles
    std::vector<uint8_t*> wl;        // per layer: the four projection matrices (bf16 or 4-bit tiles)

    __nv_bfloat16* kv = nullptr;
    float* x = nullptr;
    __nv_bfloat16 *xn = nullptr, *q = nullptr, *attn = nullptr, *h = nullptr;
    float* sq = nullptr;      // RMSNorm statistics [d/128][tokens]
    float* theta = nullptr;   // RoPE frequencies [hd/2]
    float *lmp = nullptr, *zcur = nullptr, *conf = nullptr, *tokconf = nullptr;
    int *cur = nullptr, *x0 = nullptr;
    float* chain_part = nullptr;
    int* trk = nullptr;
    int* scr_merge = nullptr;
    __nv_bfloat16* scr_side = nullptr;
    __nv_bfloat16* sls_x = nullptr;  // compacted LM-head rows
    float* sls_sq = nullptr;
    int *sls_cur = nullptr, *sls_map = nullptr, *sls_n = nullptr;
    int *chain_cnt = nullptr, *chain_done = nullptr, *epoch = nullptr;
    int *tok = nullptr, *stok = nullptr, *seq_kv = nullptr, *plan = nullptr, *outs = nullptr, *status = nullptr;
    uint8_t *st = nullptr, *sst = nullptr;
    float* logits = nullptr;  // debug, separate allocation
    size_t logits_cap = 0;
    // request mirror
    dllm_sched sched{};
    bool started = false, have_block = false;
    int B = 0, Lp = 0, gen_len = 0, n_pos = 0, kv_len = 0;
    int blk = -1, c0 = 0, c1 = 0, step = 0;
    int last_w0 = 0, last_T = 0, last_spec = 0;
    int debug = 0;
    // captured steps, one per (window rows, batch, planned cache length, debug key); all of them
    // bake in the request's schedule, so a request with another schedule drops them
    struct StepGraph {
        cudaGraphExec_t exec = nullptr;
        int T = -1, B = -1, kv = -1, dbg = -1;
        unsigned long long used = 0;  // last use, for eviction
        int n_marks = 0, launches = 0, trace_launches = 0;
        std::vector<int> ev_kind;     // the profiling events' kinds as recorded at capture
    };
    std::vector<StepGraph> graphs;
    unsigned long long graph_clock = 0;
    // per-kernel timing (events recorded after every launch of the step)
    bool profiling = false;
    std::vector<cudaEvent_t> ev;
    std::vector<int> ev_kind;
    int n_marks = 0;
    double prof_ms[DLLM_NKINDS] = {};
    int prof_launches[DLLM_NKINDS] = {};
    int prof_steps = 0;
    int launches_per_step = 0;
    bool capturing = false;
    bool in_step = false;
    // GEMM timelines of one step (debug flag 16): [launch][256 CTAs][16] stamps
    unsigned long long* trace = nullptr;
    int trace_launch = 0;
    bool poisoned = false;
    std::string err;
};

// Start of a projection matrix of layer l at offset off (elements of bf16 weights, bytes of
// 4-bit tiles).
static const void* wmat(const dllm_ctx* ctx, int l, size_t off) {
    return ctx->wl[l] + off * (ctx->L.q4 ? 1 : 2);
}

// Record a timing event after a launch of the given kind (or the start mark).
static void mark(dllm_ctx* ctx, int kind) {
    if (!ctx->in_step) return;
    if (kind >= 0) ctx->launches_per_step++;
    if (!ctx->profiling || ctx->n_marks >= static_cast<int>(ctx->ev.size())) return;
    cudaEventRecordWithFlags(ctx->ev[ctx->n_marks], ctx->stream,
                             ctx->capturing ? cudaEventRecordExternal : cudaEventRecordDefault);
    ctx->ev_kind[ctx->n_marks] = kind;
    ctx->n_marks++;
}

constexpr int kTraceLaunches = 512;
constexpr size_t kMaxStepGraphs = 32;  // captured steps kept per context (LRU)
constexpr size_t kTraceStride = 256 * 16;  // per launch: 256 CTAs x 16 slots

// Trace buffer for the GEMM launch about to be made in a step (null when off).
static unsigned long long* next_trace(dllm_ctx* ctx) {
    if (!ctx->trace || !ctx->in_step || ctx->trace_launch >= kTraceLaunches) return nullptr;
    return ctx->trace + static_cast<size_t>(ctx->trace_launch++) * kTraceStride;
}

static std::string g_noctx_err;

void dllm_set_noctx_error(const char* msg) { g_noctx_err = msg; }

static int fail(dllm_ctx* c, int code, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    if (c) {
        c->err = buf;
        if (code != DLLM_EINVAL && code != DLLM_ECAPACITY) c->poisoned = true;
    } else {
        g_noctx_err = buf;
    }
    return code;
}

#define CK(call)                                                                                   \
    do {                                                                                           \
        cudaError_t e_ = (call);                                                                   \
        if (e_ != cudaSuccess) return fail(ctx, DLLM_ECUDA, "%s: %s", #call, cudaGetErrorString(e_)); \
    } while (0)

#define GUARD(ctx)                                                         \
    do {                                                                   \
        if (!(ctx)) return fail(nullptr, DLLM_EINVAL, "null context");     \
        if ((ctx)->poisoned) return DLLM_ESTATE;                           \
    } while (0)

static int sync_check(dllm_ctx* ctx) {
    CK(cudaStreamSynchronize(ctx->stream));
    int s = 0;
    CK(cudaMemcpy(&s, ctx->status, 4, cudaMemcpyDeviceToHost));
    if (s & kStatusTimeout) return fail(ctx, DLLM_ETIMEOUT, "a bounded device wait ran out (status %d)", s);
    if (s) return fail(ctx, DLLM_ECUDA, "device status %d (index check failed)", s);
    return DLLM_OK;
}

// ------------------------------------------------------------------ forward
// Layers (and optionally the LM head) over T window tokens of each of the B
// sequences; token ids come from the state at seq_kv[b] + t.
// T window rows per sequence, then (sparse cache refresh) R tracked prefix rows:
// they run through every projection and the head, attend as queries only, and their K/V go to
// the side buffers.  With `sls` (selective logits skipping) the LM head runs as its own launch
// over the compacted rows that need a decision; the other rows get x0 = -1, conf = tokconf = 0.
// The cache length the step's attention is planned for: with sliding the frontier moves every
// few steps, so the plan (and the captured step) covers it rounded up to 64 positions; the
// kernels read each sequence's own length at run time and leave the rest of a split empty.
static int plan_kv(const dllm_ctx* ctx) {
    return ctx->sched.slide && ctx->sched.use_prefix_cache ? rup(ctx->kv_len, 64) : ctx->kv_len;
}

static int forward(dllm_ctx* ctx, int B, int Tw, bool head, int R = 0, bool sls = false) {
    const int T = Tw + R;  // rows per sequence
    const dllm_config& c = ctx->cfg;
    const Layout& L = ctx->L;
    const int d = c.d_model, F = c.ffn, qd = L.qd, N = B * T;
    cudaStream_t s = ctx->stream;
    // x = embedding rows, xb = bf16(x) (the next projection's operand), sq = RMSNorm statistics;
    // the step counter advances (it tags the chained projections' completion flags)
    CK(launch_embed(ctx->tok, c.max_ctx, ctx->seq_kv, ctx->emb, ctx->x, ctx->xn, ctx->sq, ctx->cur, ctx->epoch, B, T,
                    d, s, Tw, ctx->trk));
    mark(ctx, DLLM_K_EMBED);
    const GemmPlan pq = gemm_plan(L.qkv_rows, N, d, ctx->sms, EPI_QKV);
    const GemmPlan po = gemm_plan(L.o_rows, N, qd, ctx->sms, EPI_RESID);
    const GemmPlan pg = gemm_plan(L.gu_rows, N, d, ctx->sms, EPI_SWIGLU);
    const GemmPlan pd = gemm_plan(L.d_rows, N, F, ctx->sms, EPI_RESID);
    const GemmPlan ph = gemm_plan(L.head_rows, N, d, ctx->sms, EPI_LMHEAD);
    CUtensorMap tx_xn, tx_attn, tx_h, tx_c;
    if (!make_tmap_bf16(&tx_xn, ctx->xn, N, d, pq.ntile) || !make_tmap_bf16(&tx_attn, ctx->attn, N, qd, po.ntile) ||
        !make_tmap_bf16(&tx_h, ctx->h, N, F, pd.ntile) || !make_tmap_bf16(&tx_c, ctx->sls_x, N, d, ph.ntile))
        return fail(ctx, DLLM_ECUDA, "tensor map encode failed");
    sls = sls && head;
    AttnPlan ap = attn_plan(B, T, c.n_heads, c.head_dim, (ctx->in_step ? plan_kv(ctx) : ctx->kv_len) + Tw, ctx->sms);
    ap.qx = R;
    EpiArgs ep{};
    ep.seq_kv = ctx->seq_kv;
    ep.n_seq = B;
    ep.theta = ctx->theta;
    ep.T = T;
    ep.Tw = Tw;
    ep.R = R;
    ep.trk = ctx->trk;
    ep.H = c.n_heads;
    ep.Hkv = L.Hkv;
    ep.v_row0 = qd + L.kvd;
    ep.hd = c.head_dim;
    ep.cap = c.max_ctx;
    ep.q = ctx->q;
    ep.h = ctx->h;
    ep.F = F;
    ep.sq_in = ctx->sq;  // consumers of the residual stream apply RMSNorm as a per-token scale
    ep.n_sq = L.n_sq;
    ep.norm_dim = d;
    ep.eps = c.rms_eps;
    EpiArgs er{};
    er.out = ctx->x;
    er.ld_out = d;
    er.xb = ctx->xn;
    er.sq_out = ctx->sq;
    EpiArgs eh = ep;
    eh.lm_part = ctx->lmp;
    eh.zcur = ctx->zcur;
    eh.cur_tok = ctx->cur;
    eh.V = c.vocab;
    eh.mask_id = c.mask_id;
    eh.logits = (ctx->debug & 1) ? ctx->logits : nullptr;
    auto qkv_args = [&](int l) {
        EpiArgs e = ep;
        e.kc = ctx->kv + static_cast<size_t>(2 * l) * L.kv_half;
        e.vc = ctx->kv + static_cast<size_t>(2 * l + 1) * L.kv_half;
        e.kside = ctx->scr_side + static_cast<size_t>(2 * l) * B * L.kvd * R;  // [L][2][B][Hkv][R][hd]
        e.vside = e.kside + static_cast<size_t>(B) * L.kvd * R;
        return e;
    };
    // phase slot i of a chain uses scratch slot i; consecutive chains are ordered by the stream
    auto add_phase = [&](ChainArgs& ca, ChainMaps& m, const GemmPlan& p, int epi, EpiArgs e, int dep_rows,
                         const void* w_tiles, const CUtensorMap& x) {
        const int i = ca.n_phases++;
        ChainPhase& P = ca.ph[i];
        P.p = p;
        P.epi = epi;
        e.trace = next_trace(ctx);
        P.ep = e;
        P.dep_rows = dep_rows;
        P.partials = ctx->chain_part + static_cast<size_t>(i) * L.part_floats;
        P.tickets = ctx->chain_cnt + static_cast<size_t>(i) * L.cnt_len;
        P.done = ctx->chain_done + static_cast<size_t>(i) * L.done_len;
        P.done2 = epi == EPI_RESID ? ctx->chain_done + static_cast<size_t>(kMaxPhases + i) * L.done_len : nullptr;
        P.w_tiles = w_tiles;
        m.x[i] = x;
    };
    const int smem_budget = (ctx->debug & 8) ? kChainSmemFull : kChainSmemShared;
    auto run_chain = [&](ChainArgs& ca, const ChainMaps& m, int tag_add, int kind) -> int {
        ca.q4 = L.q4 ? 1 : 0;
        ca.epoch = ctx->epoch;
        ca.tag_mul = c.n_layers + 2;
        ca.tag_add = tag_add;
        ca.status = ctx->status;
        if (!chain_plan(ca, smem_budget)) return fail(ctx, DLLM_ECAPACITY, "projection chain does not fit");
        CK(chain_launch(m, ca, s, true));
        mark(ctx, kind);
        return DLLM_OK;
    };
    {
        ChainArgs ca{};
        ChainMaps m{};
        add_phase(ca, m, pq, EPI_QKV, qkv_args(0), 0, wmat(ctx, 0, L.w_qkv), tx_xn);
        // debug flag 32 (the bounded-wait test): this launch waits for a word nobody writes
        if ((ctx->debug & 32) && ctx->in_step) ca.gate = ctx->status + 2;
        if (int rc = run_chain(ca, m, 1, DLLM_K_QKV)) return rc;
    }
    for (int l = 0; l < c.n_layers; ++l) {
        const EpiArgs el = qkv_args(l);
        // The mma.sync attention starts per (sequence, head) on the QKV tiles it reads: layer 0's
        // come from the QKV chain (phase slot 0, tag 1), layer l's from phase slot 3 of layer
        // l-1's chain (tag l + 1).
        AttnSync sy{};
        if (!ap.tc) {
            sy.qkv_done = ctx->chain_done + static_cast<size_t>(l == 0 ? 0 : 3) * L.done_len;
            sy.qkv_ntile = pq.ntile;
            sy.qkv_ntiles = pq.n_tiles;
            sy.k_row0 = qd;
            sy.v_row0 = qd + L.kvd;
            sy.epoch = ctx->epoch;
            sy.tag_mul = c.n_layers + 2;
            sy.tag_add = l + 1;
        }
        CK(launch_attention(ctx->q, el.kc, el.vc, ctx->seq_kv, ctx->attn, B, T, c.n_heads, L.Hkv, c.head_dim, c.max_ctx,
                            ap, s, true, next_trace(ctx), ctx->status, &sy));
        mark(ctx, DLLM_K_ATTN);
        // output projection (+ residual) -> gate/up (+ SwiGLU) -> down (+ residual) -> next QKV or LM head
        ChainArgs ca{};
        ChainMaps m{};
        add_phase(ca, m, po, EPI_RESID, er, 0, wmat(ctx, l, L.w_o), tx_attn);
        add_phase(ca, m, pg, EPI_SWIGLU, ep, 128, wmat(ctx, l, L.w_gu), tx_xn);
        add_phase(ca, m, pd, EPI_RESID, er, 64, wmat(ctx, l, L.w_d), tx_h);
        if (l + 1 < c.n_layers) add_phase(ca, m, pq, EPI_QKV, qkv_args(l + 1), 128, wmat(ctx, l + 1, L.w_qkv), tx_xn);
        else if (head && !sls) add_phase(ca, m, ph, EPI_LMHEAD, eh, 128, ctx->head, tx_xn);
        if (int rc = run_chain(ca, m, l + 2, DLLM_K_LAYER)) return rc;
    }
    if (sls) {
        CK(launch_sls_map(ctx->st, c.max_ctx, ctx->seq_kv, ctx->sched.use_prefix_cache, B, Tw, T, ctx->sls_map,
                          ctx->sls_n, ctx->x0, ctx->conf, ctx->tokconf, s));
        mark(ctx, DLLM_K_HEAD);
        CK(launch_sls_gather(ctx->sls_map, ctx->sls_n, N, ph.ntile, d, ctx->xn, ctx->sq, L.n_sq, ctx->cur, ctx->sls_x,
                             ctx->sls_sq, ctx->sls_cur, s));
        mark(ctx, DLLM_K_HEAD);
        EpiArgs ec = eh;
        ec.sq_in = ctx->sls_sq;
        ec.cur_tok = ctx->sls_cur;
        ec.logits = nullptr;
        ChainArgs ca{};
        ChainMaps m{};
        add_phase(ca, m, ph, EPI_LMHEAD, ec, 0, ctx->head, tx_c);
        ca.dyn_rows = ctx->sls_n;  // the head covers only the token tiles holding the listed rows
        if (int rc = run_chain(ca, m, c.n_layers + 2, DLLM_K_HEAD)) return rc;
    }
    if (head) {
        CK(launch_lmhead_reduce(ctx->lmp, ctx->zcur, sls ? ctx->sls_cur : ctx->cur, L.head_tiles, N, c.mask_id,
                                ctx->x0, ctx->conf, ctx->tokconf, s, true, sls ? ctx->sls_map : nullptr,
                                sls ? ctx->sls_n : nullptr));
        mark(ctx, DLLM_K_HEAD_REDUCE);
    }
    return DLLM_OK;
}

static int step_kernels(dllm_ctx* ctx, int T) {
    ctx->n_marks = 0;
    ctx->launches_per_step = 0;
    ctx->trace_launch = 0;
    ctx->in_step = true;
    mark(ctx, -1);
    const int R = ctx->sched.use_prefix_cache ? ctx->sched.scr_rows : 0;
    if (R > 0) {  // the visible prefix positions this step refreshes
        CK(launch_scr_select(ctx->st, ctx->cfg.max_ctx, ctx->seq_kv, ctx->trk, ctx->B, R, ctx->stream));
        mark(ctx, DLLM_K_COMMIT);
    }
    int rc = forward(ctx, ctx->B, T, true, R, ctx->sched.sls && !(ctx->debug & 1));
    if (rc) {
        ctx->in_step = false;
        return rc;
    }
    CommitArgs a{};
    a.tok = ctx->tok;
    a.st = ctx->st;
    a.ld = ctx->cfg.max_ctx;
    a.seq_kv = ctx->seq_kv;
    a.plan = ctx->plan;
    a.x0 = ctx->x0;
    a.conf = ctx->conf;
    a.tokconf = ctx->tokconf;
    a.outs = ctx->outs;
    a.B = ctx->B;
    a.T = T;
    a.Tq = T + R;
    a.R = R;
    a.trk = ctx->trk;
    a.merge = ctx->scr_merge;
    a.mask_id = ctx->cfg.mask_id;
    a.use_cache = ctx->sched.use_prefix_cache;
    a.S = ctx->sched.steps_per_block;
    a.remask_max = ctx->sched.remask_max;
    a.spec_blocks = ctx->sched.spec_blocks;
    a.block_len = ctx->cfg.block_len;
    a.theta_remask = ctx->sched.theta_remask;
    a.theta_stable = ctx->sched.theta_stable;
    a.commit_mode = ctx->sched.commit_mode;
    a.slide_kv = ctx->sched.slide && ctx->sched.use_prefix_cache ? ctx->seq_kv : nullptr;
    a.theta_visible = ctx->sched.theta_visible;
    cudaError_t ce = launch_commit(a, ctx->stream);
    mark(ctx, DLLM_K_COMMIT);
    if (ce == cudaSuccess && R > 0) {  // the refreshed K/V merged at the step boundary
        ce = launch_scr_merge(ctx->scr_side, ctx->kv, ctx->trk, ctx->scr_merge, ctx->cfg.n_layers, ctx->B,
                              ctx->cfg.max_batch, ctx->L.Hkv, ctx->cfg.head_dim, ctx->cfg.max_ctx, R,
                              ctx->stream);
        mark(ctx, DLLM_K_COMMIT);
    }
    ctx->in_step = false;
    CK(ce);
    return DLLM_OK;
}

static int profile_collect(dllm_ctx* ctx) {
    if (!ctx->profiling || ctx->n_marks < 2) return DLLM_OK;
    CK(cudaStreamSynchronize(ctx->stream));
    int launches[DLLM_NKINDS] = {};
    for (int i = 1; i < ctx->n_marks; ++i) {
        float ms = 0.0f;
        CK(cudaEventElapsedTime(&ms, ctx->ev[i - 1], ctx->ev[i]));
        int k = ctx->ev_kind[i];
        if (k >= 0 && k < DLLM_NKINDS) {
            ctx->prof_ms[k] += ms;
            launches[k]++;
        }
    }
    for (int k = 0; k < DLLM_NKINDS; ++k) ctx->prof_launches[k] = launches[k];
    ctx->prof_steps++;
    return DLLM_OK;
}

// ------------------------------------------------------------------ ABI
extern "C" {

int dllm_arena_bytes(const dllm_config* cfg, size_t* bytes) {
    if (!cfg || !bytes) return fail(nullptr, DLLM_EINVAL, "null argument");
    if (const char* m = check_cfg(*cfg)) return fail(nullptr, DLLM_EINVAL, "%s", m);
    *bytes = make_layout(*cfg).total;
    return DLLM_OK;
}

const char* dllm_last_error(const dllm_ctx* ctx) { return ctx ? ctx->err.c_str() : g_noctx_err.c_str(); }

void dllm_free(dllm_ctx* ctx) {
    if (!ctx) return;
    if (ctx->stream) cudaStreamSynchronize(ctx->stream);
    for (auto& g : ctx->graphs) cudaGraphExecDestroy(g.exec);
    for (cudaEvent_t e : ctx->ev) cudaEventDestroy(e);
    if (ctx->logits) cudaFree(ctx->logits);
    if (ctx->trace) cudaFree(ctx->trace);
    if (ctx->own_arena && ctx->arena) cudaFree(ctx->arena);
    if (ctx->own_stream && ctx->stream) cudaStreamDestroy(ctx->stream);
    delete ctx;
}

int dllm_init(const dllm_config* cfg, void* dev_arena, size_t arena_bytes, void* cuda_stream, dllm_ctx** out) {
    if (!cfg || !out) return fail(nullptr, DLLM_EINVAL, "null argument");
    *out = nullptr;
    if (const char* m = check_cfg(*cfg)) return fail(nullptr, DLLM_EINVAL, "%s", m);
    dllm_ctx* ctx = new (std::nothrow) dllm_ctx();
    if (!ctx) return fail(nullptr, DLLM_ENOMEM, "host allocation failed");
    ctx->cfg = *cfg;
    ctx->L = make_layout(*cfg);
    const Layout& L = ctx->L;
    const dllm_config& c = ctx->cfg;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&ctx->sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) {
        int rc = fail(nullptr, DLLM_ECUDA, "no CUDA device: %s", cudaGetErrorString(e));
        delete ctx;
        return rc;
    }
    ctx->sms = std::min(ctx->sms, kMaxSMs);
    auto bail = [&](int code, const char* msg) {
        g_noctx_err = msg;
        dllm_free(ctx);
        return code;
    };
    if (cuda_stream) {
        ctx->stream = static_cast<cudaStream_t>(cuda_stream);
    } else {
        if (cudaStreamCreateWithFlags(&ctx->stream, cudaStreamNonBlocking) != cudaSuccess)
            return bail(DLLM_ECUDA, "stream creation failed");
        ctx->own_stream = true;
    }
    if (dev_arena) {
        if (arena_bytes < L.total || (reinterpret_cast<uintptr_t>(dev_arena) & 255))
            return bail(DLLM_EINVAL, "arena too small or not 256-byte aligned");
        ctx->arena = static_cast<uint8_t*>(dev_arena);
    } else {
        if (cudaMalloc(&ctx->arena, L.total) != cudaSuccess) return bail(DLLM_ENOMEM, "device allocation failed");
        ctx->own_arena = true;
    }
    if (gemm_init_attrs() != cudaSuccess || attn_init_attrs() != cudaSuccess || chain_init_attrs() != cudaSuccess)
        return bail(DLLM_ECUDA, "kernel attribute setup failed");
    uint8_t* A = ctx->arena;
    const int d = c.d_model, F = c.ffn, qd = L.qd;
    ctx->emb = reinterpret_cast<__nv_bfloat16*>(A + L.off_emb);
    ctx->head = A + L.off_head;
    ctx->kv = reinterpret_cast<__nv_bfloat16*>(A + L.off_kv);
    ctx->x = reinterpret_cast<float*>(A + L.off_x);
    ctx->xn = reinterpret_cast<__nv_bfloat16*>(A + L.off_xn);
    ctx->q = reinterpret_cast<__nv_bfloat16*>(A + L.off_q);
    ctx->attn = reinterpret_cast<__nv_bfloat16*>(A + L.off_attn);
    ctx->h = reinterpret_cast<__nv_bfloat16*>(A + L.off_h);
    ctx->sq = reinterpret_cast<float*>(A + L.off_sq);
    ctx->theta = reinterpret_cast<float*>(A + L.off_theta);
    ctx->lmp = reinterpret_cast<float*>(A + L.off_lmp);
    ctx->zcur = reinterpret_cast<float*>(A + L.off_zcur);
    ctx->cur = reinterpret_cast<int*>(A + L.off_cur);
    ctx->x0 = reinterpret_cast<int*>(A + L.off_x0);
    ctx->conf = reinterpret_cast<float*>(A + L.off_conf);
    ctx->tokconf = reinterpret_cast<float*>(A + L.off_tokconf);
    ctx->chain_part = reinterpret_cast<float*>(A + L.off_part);
    ctx->chain_cnt = reinterpret_cast<int*>(A + L.off_cnt);
    ctx->chain_done = reinterpret_cast<int*>(A + L.off_done);
    ctx->epoch = reinterpret_cast<int*>(A + L.off_epoch);
    ctx->tok = reinterpret_cast<int*>(A + L.off_tok);
    ctx->st = A + L.off_st;
    ctx->stok = reinterpret_cast<int*>(A + L.off_stok);
    ctx->sst = A + L.off_sst;
    ctx->seq_kv = reinterpret_cast<int*>(A + L.off_seqkv);
    ctx->plan = reinterpret_cast<int*>(A + L.off_plan);
    ctx->outs = reinterpret_cast<int*>(A + L.off_outs);
    ctx->status = reinterpret_cast<int*>(A + L.off_status);
    ctx->trk = reinterpret_cast<int*>(A + L.off_trk);
    ctx->scr_merge = reinterpret_cast<int*>(A + L.off_smerge);
    ctx->scr_side = reinterpret_cast<__nv_bfloat16*>(A + L.off_side);
    ctx->sls_x = reinterpret_cast<__nv_bfloat16*>(A + L.off_xc);
    ctx->sls_sq = reinterpret_cast<float*>(A + L.off_sqc);
    ctx->sls_cur = reinterpret_cast<int*>(A + L.off_curc);
    ctx->sls_map = reinterpret_cast<int*>(A + L.off_rmap);
    ctx->sls_n = reinterpret_cast<int*>(A + L.off_nrows);
    cudaStream_t s = ctx->stream;
    // zero everything that is read before it is written (counters, state, status)
    if (cudaMemsetAsync(A + L.off_sq, 0, L.total - L.off_sq, s) != cudaSuccess ||
        cudaMemsetAsync(A + L.off_kv, 0, L.kv_half * 4 * c.n_layers, s) != cudaSuccess)
        return bail(DLLM_ECUDA, "memset failed");
    // weights from the seed (tensor ids: embedding 1, head 2, layer l: 16 + 8l + {q,k,v,o,gate,up,down})
    const uint64_t seed = c.weight_seed;
    const int hd = c.head_dim;
    // (the embedding is gathered by rows: row-major; the projections are streamed: tile-major)
    const int kvd = L.kvd;
    // a projection matrix (rows_phys x cols, row order `mode`) of tensors tid.. in the context's format
    auto init_w = [&](uint8_t* dst, int mode, int rows_phys, int cols, int logical_rows, uint64_t tid) {
        return L.q4 ? launch_init_weight_q4(dst, mode, rows_phys, cols, logical_rows, seed, tid, qd, kvd, hd, s)
                    : launch_init_weight(reinterpret_cast<__nv_bfloat16*>(dst), mode, rows_phys, cols, logical_rows,
                                         seed, tid, qd, kvd, hd, true, s);
    };
    cudaError_t ie = launch_init_weight(ctx->emb, 0, c.vocab, d, c.vocab, seed, 1, qd, kvd, hd, false, s);
    if (ie == cudaSuccess) ie = init_w(ctx->head, 0, L.head_rows, d, c.vocab, 2);
    ctx->wl.resize(c.n_layers);
    const size_t unit = L.q4 ? 1 : 2;  // bytes per layout offset unit
    for (int l = 0; l < c.n_layers && ie == cudaSuccess; ++l) {
        uint8_t* w = A + L.off_w + static_cast<size_t>(l) * L.per_layer * unit;
        ctx->wl[l] = w;
        const uint64_t t0 = 16 + 8ull * l;
        ie = init_w(w + L.w_qkv * unit, 1, L.qkv_rows, d, qd, t0 + 0);
        if (ie == cudaSuccess) ie = init_w(w + L.w_o * unit, 0, L.o_rows, qd, d, t0 + 3);
        if (ie == cudaSuccess) ie = init_w(w + L.w_gu * unit, 2, L.gu_rows, d, F, t0 + 4);
        if (ie == cudaSuccess) ie = init_w(w + L.w_d * unit, 0, L.d_rows, F, d, t0 + 6);
    }
    // RoPE frequencies base^(-2j/hd), in double on the host
    std::vector<float> th(c.head_dim / 2);
    for (int j = 0; j < c.head_dim / 2; ++j)
        th[j] = static_cast<float>(std::pow(static_cast<double>(c.rope_base), -2.0 * j / c.head_dim));
    if (ie == cudaSuccess) ie = cudaMemcpyAsync(ctx->theta, th.data(), th.size() * 4, cudaMemcpyHostToDevice, s);
    if (ie != cudaSuccess || cudaStreamSynchronize(s) != cudaSuccess) return bail(DLLM_ECUDA, "weight init failed");
    *out = ctx;
    return DLLM_OK;
}

int dllm_sync(dllm_ctx* ctx) {
    GUARD(ctx);
    return sync_check(ctx);
}

static int set_debug_buffers(dllm_ctx* ctx) {
    if ((ctx->debug & 16) && !ctx->trace) {
        if (cudaMalloc(&ctx->trace, kTraceLaunches * kTraceStride * 8) != cudaSuccess)
            return fail(ctx, DLLM_ENOMEM, "trace buffer");
        cudaMemset(ctx->trace, 0, kTraceLaunches * kTraceStride * 8);
    }
    if (!(ctx->debug & 1)) return DLLM_OK;
    size_t need = static_cast<size_t>(ctx->L.max_tok) * ctx->cfg.vocab;
    if (ctx->logits_cap >= need) return DLLM_OK;
    if (ctx->logits) cudaFree(ctx->logits);
    if (ctx->trace) cudaFree(ctx->trace);
    ctx->logits = nullptr;
    if (cudaMalloc(&ctx->logits, need * 4) != cudaSuccess) return fail(ctx, DLLM_ENOMEM, "logits buffer");
    ctx->logits_cap = need;
    return DLLM_OK;
}

int dllm_set_debug(dllm_ctx* ctx, int flags) {
    GUARD(ctx);
    ctx->debug = flags;
    set_pdl(!(flags & 4));
    set_stream_smem(!(flags & 8));
    return set_debug_buffers(ctx);
}

static int start_request(dllm_ctx* ctx, const dllm_sched* sched, int batch, int Lp, int gen_len,
                         const int32_t* prompt, int P_random, uint64_t kv_seed) {
    const dllm_config& c = ctx->cfg;
    if (!sched || batch < 1 || Lp < 0 || gen_len < 1) return fail(ctx, DLLM_EINVAL, "bad request arguments");
    if (sched->steps_per_block < 1 || sched->remask_max < 0 || sched->spec_blocks < 0 ||
        (sched->commit_mode != DLLM_COMMIT_SCHEDULE && sched->commit_mode != DLLM_COMMIT_THRESHOLD) ||
        !(sched->theta_visible == sched->theta_visible) || sched->scr_rows < 0 ||
        sched->scr_rows > DLLM_MAX_SCR_ROWS || sched->spec_lat_n < 0 || sched->spec_lat_n > 8 ||
        (sched->sls != 0 && sched->sls != 1) || (sched->slide != 0 && sched->slide != 1))
        return fail(ctx, DLLM_EINVAL, "bad schedule");
    if (sched->scr_rows > 0 && !sched->use_prefix_cache)
        return fail(ctx, DLLM_EINVAL, "sparse cache refresh needs the prefix cache");
    if (sched->slide && (!sched->use_prefix_cache || batch != 1))
        return fail(ctx, DLLM_EINVAL, "continuous sliding needs the prefix cache and batch 1");
    if (sched->use_prefix_cache && c.block_len * (1 + sched->spec_blocks) + sched->scr_rows > c.max_window)
        return fail(ctx, DLLM_ECAPACITY, "window plus refresh rows > max_window %d", c.max_window);
    if (batch > c.max_batch) return fail(ctx, DLLM_ECAPACITY, "batch %d > max_batch %d", batch, c.max_batch);
    const int n_pos = Lp + gen_len;
    if (n_pos > c.max_ctx) return fail(ctx, DLLM_ECAPACITY, "Lp + gen_len = %d > max_ctx %d", n_pos, c.max_ctx);
    int maxT = sched->use_prefix_cache ? std::max(P_random ? 0 : Lp, c.block_len * (1 + sched->spec_blocks)) : n_pos;
    if (maxT > c.max_window) return fail(ctx, DLLM_ECAPACITY, "window of %d tokens > max_window %d", maxT, c.max_window);
    if (!sched->use_prefix_cache && gen_len > kMaxBlock) return fail(ctx, DLLM_ECAPACITY, "block too long");
    if (prompt)
        for (int b = 0; b < batch; ++b)
            for (int p = 0; p < Lp; ++p) {
                int v = prompt[static_cast<size_t>(b) * Lp + p];
                if (v < 0 || v >= c.vocab) return fail(ctx, DLLM_EINVAL, "prompt id %d out of range", v);
            }
    if (memcmp(&ctx->sched, sched, sizeof(dllm_sched)) != 0) {
        // the captured steps bake in the schedule's thresholds and counts
        for (auto& g : ctx->graphs) cudaGraphExecDestroy(g.exec);
        ctx->graphs.clear();
    }
    ctx->sched = *sched;
    ctx->B = batch;
    ctx->Lp = Lp;
    ctx->gen_len = gen_len;
    ctx->n_pos = n_pos;
    ctx->blk = -1;
    ctx->have_block = false;
    ctx->started = false;
    ctx->step = 0;
    ctx->kv_len = 0;
    // state rows
    std::vector<int32_t> tok(static_cast<size_t>(batch) * c.max_ctx, c.mask_id);
    std::vector<uint8_t> st(static_cast<size_t>(batch) * c.max_ctx, DLLM_MASKED);
    for (int b = 0; b < batch; ++b)
        for (int p = 0; p < Lp; ++p) {
            tok[static_cast<size_t>(b) * c.max_ctx + p] = prompt ? prompt[static_cast<size_t>(b) * Lp + p] : 0;
            st[static_cast<size_t>(b) * c.max_ctx + p] = DLLM_FIXED;
        }
    CK(cudaMemcpyAsync(ctx->tok, tok.data(), tok.size() * 4, cudaMemcpyHostToDevice, ctx->stream));
    CK(cudaMemcpyAsync(ctx->st, st.data(), st.size(), cudaMemcpyHostToDevice, ctx->stream));
    CK(launch_set_kv_len(ctx->seq_kv, batch, 0, ctx->stream));
    CK(cudaStreamSynchronize(ctx->stream));  // host vectors go out of scope
    if (P_random) {
        for (int l = 0; l < c.n_layers; ++l)
            for (int w = 0; w < 2; ++w)
                CK(launch_init_kv_random(ctx->kv + static_cast<size_t>(2 * l + w) * ctx->L.kv_half, batch, ctx->L.Hkv,
                                         c.head_dim, c.max_ctx, Lp, l, w, c.n_layers, kv_seed, ctx->stream));
        ctx->kv_len = Lp;
        CK(launch_set_kv_len(ctx->seq_kv, batch, Lp, ctx->stream));
    } else if (sched->use_prefix_cache && Lp > 0) {
        int rc = forward(ctx, batch, Lp, false);
        if (rc) return rc;
        ctx->kv_len = Lp;
        CK(launch_set_kv_len(ctx->seq_kv, batch, Lp, ctx->stream));
    }
    ctx->started = true;
    return sync_check(ctx);
}

int dllm_prefill(dllm_ctx* ctx, const dllm_sched* sched, int batch, const int32_t* prompt, int Lp, int gen_len) {
    GUARD(ctx);
    if (!prompt && Lp > 0) return fail(ctx, DLLM_EINVAL, "null prompt");
    return start_request(ctx, sched, batch, Lp, gen_len, prompt, 0, 0);
}

int dllm_set_prefix_kv_random(dllm_ctx* ctx, const dllm_sched* sched, int batch, int P, int gen_len, uint64_t seed) {
    GUARD(ctx);
    if (!sched || !sched->use_prefix_cache || P < 1) return fail(ctx, DLLM_EINVAL, "synthetic prefix needs the cache");
    return start_request(ctx, sched, batch, P, gen_len, nullptr, 1, seed);
}

static int count_masked_max(dllm_ctx* ctx, int a, int b, int* out) {
    const int ld = ctx->cfg.max_ctx;
    std::vector<uint8_t> st(static_cast<size_t>(ctx->B) * ld);
    CK(cudaMemcpyAsync(st.data(), ctx->st, st.size(), cudaMemcpyDeviceToHost, ctx->stream));
    int rc = sync_check(ctx);
    if (rc) return rc;
    int mx = 0;
    for (int s = 0; s < ctx->B; ++s) {
        int m = 0;
        for (int p = a; p < b; ++p) m += st[static_cast<size_t>(s) * ld + p] == DLLM_MASKED;
        mx = std::max(mx, m);
    }
    *out = mx;
    return DLLM_OK;
}

int dllm_begin_block(dllm_ctx* ctx) {
    GUARD(ctx);
    if (!ctx->started) return fail(ctx, DLLM_EINVAL, "no request: call dllm_prefill first");
    const dllm_config& c = ctx->cfg;
    if (ctx->have_block) {
        int m = 0;
        int rc = count_masked_max(ctx, ctx->c0, ctx->c1, &m);
        if (rc) return rc;
        if (m) return fail(ctx, DLLM_EINVAL, "current block still has %d masked positions", m);
        if (ctx->sched.use_prefix_cache) {
            // recompute the finished block's K/V from its final ids and append them (with
            // sliding: the part that has not slid into the cache yet)
            const int rem = ctx->c1 - ctx->kv_len;
            if (rem > 0) {
                rc = forward(ctx, ctx->B, rem, false);
                if (rc) return rc;
            }
            ctx->kv_len = ctx->c1;
            CK(launch_set_kv_len(ctx->seq_kv, ctx->B, ctx->kv_len, ctx->stream));
        }
        ctx->have_block = false;
    }
    const int bl = ctx->sched.use_prefix_cache ? c.block_len : c.block_len;
    int nb = ctx->blk + 1;
    int c0 = ctx->Lp + nb * bl;
    if (c0 >= ctx->n_pos) {
        ctx->blk = nb;
        int rc = sync_check(ctx);
        return rc ? rc : DLLM_DONE;
    }
    ctx->blk = nb;
    ctx->c0 = c0;
    ctx->c1 = std::min(c0 + bl, ctx->n_pos);
    ctx->step = 0;
    CK(launch_begin_block(ctx->tok, ctx->st, ctx->stok, ctx->sst, c.max_ctx, ctx->n_pos, ctx->plan, ctx->B, ctx->c0,
                          ctx->c1, ctx->stream));
    ctx->have_block = true;
    return DLLM_OK;
}

int dllm_rewind_block(dllm_ctx* ctx) {
    GUARD(ctx);
    if (!ctx->have_block) return fail(ctx, DLLM_EINVAL, "no current block");
    CK(launch_rewind(ctx->tok, ctx->st, ctx->stok, ctx->sst, ctx->cfg.max_ctx, ctx->n_pos, ctx->plan, ctx->B,
                     ctx->stream));
    if (ctx->sched.slide && ctx->sched.use_prefix_cache && ctx->kv_len != ctx->c0) {  // the frontier goes back too
        ctx->kv_len = ctx->c0;
        CK(launch_set_kv_len(ctx->seq_kv, ctx->B, ctx->kv_len, ctx->stream));
    }
    ctx->step = 0;
    return DLLM_OK;
}

int dllm_denoise_step(dllm_ctx* ctx, dllm_step_out* out) {
    GUARD(ctx);
    if (!ctx->have_block) return fail(ctx, DLLM_EINVAL, "no current block: call dllm_begin_block");
    const dllm_sched& s = ctx->sched;
    const int bl = ctx->cfg.block_len;
    int w0, T, spec = 0;
    if (s.use_prefix_cache) {
        w0 = ctx->kv_len;
        // the window without lookahead: the current block, or with sliding one block's length
        // from the frontier
        const int base = s.slide ? std::min(w0 + bl, ctx->n_pos) : ctx->c1;
        int w1 = base;
        if (s.spec_blocks > 0 && base < ctx->n_pos) {
            int m = 0;
            int rc = count_masked_max(ctx, ctx->c0, ctx->c1, &m);
            if (rc) return rc;
            if (m <= s.spec_trigger) {
                int k = s.spec_blocks;
                if (s.spec_allowance >= 0.0f && s.spec_lat_n > 0) {
                    // greedy: one more future block while the step stays within the allowance
                    const int i0 = (base - w0 + bl - 1) / bl - 1;
                    k = 0;
                    for (int j = 1; j <= s.spec_blocks; ++j) {
                        const int i = i0 + j;
                        if (i0 < 0 || i >= s.spec_lat_n || i0 >= s.spec_lat_n) break;
                        if (s.spec_lat[i] > (1.0f + s.spec_allowance) * s.spec_lat[i0]) break;
                        k = j;
                    }
                }
                if (k > 0) {
                    spec = 1;
                    w1 = std::min(base + k * bl, ctx->n_pos);
                }
            }
        }
        T = w1 - w0;
    } else {
        w0 = 0;
        T = ctx->n_pos;
    }
    ctx->last_w0 = w0;
    ctx->last_T = T;
    ctx->last_spec = spec;
    const bool use_graph = !(ctx->debug & 2);
    if (use_graph) {
        // trace pointers and the refresh rows are baked in too
        const int key_dbg = ctx->debug | (ctx->profiling ? 256 : 0) |
                            ((s.use_prefix_cache ? s.scr_rows : 0) << 10) | (s.sls << 16);
        const int kv = plan_kv(ctx);
        dllm_ctx::StepGraph* hit = nullptr;
        for (auto& g : ctx->graphs)
            if (g.T == T && g.B == ctx->B && g.kv == kv && g.dbg == key_dbg) hit = &g;
        if (!hit) {
            cudaGraph_t g = nullptr;
            CK(cudaStreamBeginCapture(ctx->stream, cudaStreamCaptureModeThreadLocal));
            ctx->capturing = true;
            int rc = step_kernels(ctx, T);
            ctx->capturing = false;
            cudaError_t ee = cudaStreamEndCapture(ctx->stream, &g);
            if (rc) {
                if (g) cudaGraphDestroy(g);
                return rc;
            }
            if (ee != cudaSuccess) return fail(ctx, DLLM_ECUDA, "graph capture: %s", cudaGetErrorString(ee));
            cudaGraphExec_t exec = nullptr;
            ee = cudaGraphInstantiate(&exec, g, 0);
            cudaGraphDestroy(g);
            if (ee != cudaSuccess) return fail(ctx, DLLM_ECUDA, "graph instantiate: %s", cudaGetErrorString(ee));
            if (ctx->graphs.size() >= kMaxStepGraphs) {  // evict the least recently used
                size_t lru = 0;
                for (size_t i = 1; i < ctx->graphs.size(); ++i)
                    if (ctx->graphs[i].used < ctx->graphs[lru].used) lru = i;
                cudaGraphExecDestroy(ctx->graphs[lru].exec);
                ctx->graphs.erase(ctx->graphs.begin() + static_cast<long>(lru));
            }
            dllm_ctx::StepGraph sg;
            sg.exec = exec;
            sg.T = T;
            sg.B = ctx->B;
            sg.kv = kv;
            sg.dbg = key_dbg;
            sg.n_marks = ctx->n_marks;
            sg.launches = ctx->launches_per_step;
            sg.trace_launches = ctx->trace_launch;
            sg.ev_kind = ctx->ev_kind;
            ctx->graphs.push_back(sg);
            hit = &ctx->graphs.back();
        }
        hit->used = ++ctx->graph_clock;
        // what the replayed graph records: its own events' kinds, launch and trace counts
        ctx->n_marks = hit->n_marks;
        ctx->launches_per_step = hit->launches;
        ctx->trace_launch = hit->trace_launches;
        if (!hit->ev_kind.empty()) ctx->ev_kind = hit->ev_kind;
        CK(cudaGraphLaunch(hit->exec, ctx->stream));
    } else {
        int rc = step_kernels(ctx, T);
        if (rc) return rc;
    }
    {
        int rc = profile_collect(ctx);
        if (rc) return rc;
    }
    ctx->step++;
    if (s.slide && s.use_prefix_cache) {  // the frontier the commit pass moved
        int kv = 0;
        CK(cudaMemcpyAsync(&kv, ctx->seq_kv, 4, cudaMemcpyDeviceToHost, ctx->stream));
        int rc = sync_check(ctx);
        if (rc) return rc;
        ctx->kv_len = kv;
    }
    if (out) {
        std::vector<int> o(static_cast<size_t>(ctx->B) * 8);
        CK(cudaMemcpyAsync(o.data(), ctx->outs, o.size() * 4, cudaMemcpyDeviceToHost, ctx->stream));
        int rc = sync_check(ctx);
        if (rc) return rc;
        memset(out, 0, sizeof(*out));
        out->block_done = 1;
        for (int b = 0; b < ctx->B; ++b) {
            const int* r = &o[static_cast<size_t>(b) * 8];
            out->n_committed += r[0];
            out->n_remasked += r[1];
            out->n_stable += r[2];
            out->n_drafts += r[3];
            out->block_done &= r[4];
            out->masked_after += r[5];
            out->n_refreshed += r[6];
            out->n_revised += r[7];
        }
    }
    return DLLM_OK;
}

int dllm_generate(dllm_ctx* ctx, const dllm_sched* sched, int batch, const int32_t* prompt, int Lp, int gen_len,
                  int32_t* out_tokens, dllm_stats* stats) {
    GUARD(ctx);
    int rc = dllm_prefill(ctx, sched, batch, prompt, Lp, gen_len);
    if (rc) return rc;
    dllm_stats stt{};
    // LLaDA's fixed schedule without lookahead or sliding finishes a block of at least S
    // positions in exactly S = steps_per_block steps (every step commits at least one position
    // and leaves at least one per remaining step; re-masks only add to the count; the last step
    // commits what is left): those steps are queued without a read-back, the last one reports
    const bool fixed_len = sched->commit_mode == DLLM_COMMIT_SCHEDULE && sched->spec_blocks == 0 && !sched->slide;
    while ((rc = dllm_begin_block(ctx)) == DLLM_OK) {
        dllm_step_out o{};
        if (fixed_len && sched->steps_per_block <= ctx->c1 - ctx->c0)
            for (int i = 0; i + 1 < sched->steps_per_block; ++i) {
                rc = dllm_denoise_step(ctx, nullptr);
                if (rc) return rc;
                stt.steps++;
            }
        // a block finishes within S steps (schedule), or within the revision horizon S plus one
        // step per position (threshold: every step commits at least one)
        for (int guard = 0; guard < 4 * sched->steps_per_block + 4 + ctx->cfg.block_len; ++guard) {
            rc = dllm_denoise_step(ctx, &o);
            if (rc) return rc;
            stt.steps++;
            stt.spec_steps += ctx->last_spec;
            if (o.block_done) break;
        }
        if (!o.block_done) return fail(ctx, DLLM_ESTATE, "block did not finish");
        stt.blocks++;
    }
    if (rc != DLLM_DONE) return rc;
    if (stats) *stats = stt;
    if (out_tokens) {
        const int ld = ctx->cfg.max_ctx;
        for (int b = 0; b < batch; ++b)
            CK(cudaMemcpyAsync(out_tokens + static_cast<size_t>(b) * gen_len, ctx->tok + static_cast<size_t>(b) * ld + Lp,
                               static_cast<size_t>(gen_len) * 4, cudaMemcpyDeviceToHost, ctx->stream));
    }
    return sync_check(ctx);
}

int dllm_set_profile(dllm_ctx* ctx, int enable) {
    GUARD(ctx);
    if (enable && ctx->ev.empty()) {
        const int n = 16 * ctx->cfg.n_layers + 32;
        ctx->ev.resize(n);
        ctx->ev_kind.assign(n, -1);
        for (int i = 0; i < n; ++i) CK(cudaEventCreate(&ctx->ev[i]));
    }
    ctx->profiling = enable != 0;
    for (int k = 0; k < DLLM_NKINDS; ++k) {
        ctx->prof_ms[k] = 0.0;
        ctx->prof_launches[k] = 0;
    }
    ctx->prof_steps = 0;
    return DLLM_OK;
}

int dllm_get_profile(dllm_ctx* ctx, double* ms_total, int32_t* launches_per_step, int32_t* steps) {
    GUARD(ctx);
    for (int k = 0; k < DLLM_NKINDS; ++k) {
        if (ms_total) ms_total[k] = ctx->prof_ms[k];
        if (launches_per_step) launches_per_step[k] = ctx->prof_launches[k];
    }
    if (steps) *steps = ctx->prof_steps;
    return DLLM_OK;
}

int dllm_get_trace(dllm_ctx* ctx, unsigned long long* out, int max_launches, int32_t* n_launches) {
    GUARD(ctx);
    if (!ctx->trace || !out || !n_launches) return fail(ctx, DLLM_EINVAL, "tracing needs dllm_set_debug(16)");
    const int n = ctx->trace_launch < max_launches ? ctx->trace_launch : max_launches;
    CK(cudaMemcpyAsync(out, ctx->trace, static_cast<size_t>(n) * kTraceStride * 8, cudaMemcpyDeviceToHost,
                       ctx->stream));
    *n_launches = n;
    return sync_check(ctx);
}

int dllm_launches_per_step(dllm_ctx* ctx, int32_t* n) {
    GUARD(ctx);
    if (!n) return fail(ctx, DLLM_EINVAL, "null output");
    *n = ctx->launches_per_step;
    return DLLM_OK;
}

int dllm_window(dllm_ctx* ctx, int32_t* info) {
    GUARD(ctx);
    if (!info) return fail(ctx, DLLM_EINVAL, "null info");
    info[0] = ctx->last_w0;
    info[1] = ctx->last_T;
    info[2] = ctx->c0;
    info[3] = ctx->c1;
    info[4] = ctx->step;
    info[5] = ctx->kv_len;
    info[6] = ctx->last_spec;
    return DLLM_OK;
}

int dllm_get_state(dllm_ctx* ctx, int32_t* tokens, uint8_t* status, int32_t* kv_len) {
    GUARD(ctx);
    if (!ctx->started) return fail(ctx, DLLM_EINVAL, "no request");
    const int ld = ctx->cfg.max_ctx, n = ctx->n_pos;
    for (int b = 0; b < ctx->B; ++b) {
        if (tokens)
            CK(cudaMemcpyAsync(tokens + static_cast<size_t>(b) * n, ctx->tok + static_cast<size_t>(b) * ld,
                               static_cast<size_t>(n) * 4, cudaMemcpyDeviceToHost, ctx->stream));
        if (status)
            CK(cudaMemcpyAsync(status + static_cast<size_t>(b) * n, ctx->st + static_cast<size_t>(b) * ld, n,
                               cudaMemcpyDeviceToHost, ctx->stream));
    }
    if (kv_len)
        for (int b = 0; b < ctx->B; ++b) kv_len[b] = ctx->kv_len;
    return sync_check(ctx);
}

int dllm_set_state(dllm_ctx* ctx, const int32_t* tokens, const uint8_t* status) {
    GUARD(ctx);
    if (!ctx->started) return fail(ctx, DLLM_EINVAL, "no request");
    const int ld = ctx->cfg.max_ctx, n = ctx->n_pos;
    for (int b = 0; b < ctx->B; ++b) {
        if (tokens)
            CK(cudaMemcpyAsync(ctx->tok + static_cast<size_t>(b) * ld, tokens + static_cast<size_t>(b) * n,
                               static_cast<size_t>(n) * 4, cudaMemcpyHostToDevice, ctx->stream));
        if (status)
            CK(cudaMemcpyAsync(ctx->st + static_cast<size_t>(b) * ld, status + static_cast<size_t>(b) * n, n,
                               cudaMemcpyHostToDevice, ctx->stream));
    }
    if (ctx->have_block) {  // the new state is what dllm_rewind_block returns to
        const size_t rows = static_cast<size_t>(ctx->B) * ld;
        CK(cudaMemcpyAsync(ctx->stok, ctx->tok, rows * 4, cudaMemcpyDeviceToDevice, ctx->stream));
        CK(cudaMemcpyAsync(ctx->sst, ctx->st, rows, cudaMemcpyDeviceToDevice, ctx->stream));
    }
    return sync_check(ctx);  // the caller's buffers may be reused on return
}

int dllm_get_step_debug(dllm_ctx* ctx, float* logits, int32_t* argmax, float* conf, float* tokconf) {
    GUARD(ctx);
    // a sequence's rows: its T window rows (then, with sparse cache refresh, its refresh rows)
    const size_t T = static_cast<size_t>(ctx->last_T), B = static_cast<size_t>(ctx->B);
    const size_t Tq = T + (ctx->sched.use_prefix_cache ? ctx->sched.scr_rows : 0);
    const size_t V = static_cast<size_t>(ctx->cfg.vocab);
    if (logits) {
        if (!(ctx->debug & 1) || !ctx->logits) return fail(ctx, DLLM_EINVAL, "logits need dllm_set_debug(1)");
        CK(cudaMemcpy2DAsync(logits, T * V * 4, ctx->logits, Tq * V * 4, T * V * 4, B, cudaMemcpyDeviceToHost,
                             ctx->stream));
    }
    if (argmax) CK(cudaMemcpy2DAsync(argmax, T * 4, ctx->x0, Tq * 4, T * 4, B, cudaMemcpyDeviceToHost, ctx->stream));
    if (conf) CK(cudaMemcpy2DAsync(conf, T * 4, ctx->conf, Tq * 4, T * 4, B, cudaMemcpyDeviceToHost, ctx->stream));
    if (tokconf)
        CK(cudaMemcpy2DAsync(tokconf, T * 4, ctx->tokconf, Tq * 4, T * 4, B, cudaMemcpyDeviceToHost, ctx->stream));
    return sync_check(ctx);
}

int dllm_get_scr_debug(dllm_ctx* ctx, int32_t* pos, int32_t* argmax, float* conf, float* tokconf, int* n) {
    GUARD(ctx);
    const int R = ctx->sched.use_prefix_cache ? ctx->sched.scr_rows : 0;
    if (n) *n = R;
    if (R == 0) return DLLM_OK;
    // sequence b's rows T .. T + R - 1 of its T + R
    const size_t T = static_cast<size_t>(ctx->last_T), Tq = T + R, B = static_cast<size_t>(ctx->B);
    if (pos) CK(cudaMemcpyAsync(pos, ctx->trk, B * R * 4, cudaMemcpyDeviceToHost, ctx->stream));
    if (argmax) CK(cudaMemcpy2DAsync(argmax, R * 4, ctx->x0 + T, Tq * 4, R * 4, B, cudaMemcpyDeviceToHost, ctx->stream));
    if (conf) CK(cudaMemcpy2DAsync(conf, R * 4, ctx->conf + T, Tq * 4, R * 4, B, cudaMemcpyDeviceToHost, ctx->stream));
    if (tokconf)
        CK(cudaMemcpy2DAsync(tokconf, R * 4, ctx->tokconf + T, Tq * 4, R * 4, B, cudaMemcpyDeviceToHost, ctx->stream));
    return sync_check(ctx);
}

int dllm_get_weight(dllm_ctx* ctx, int layer, int which, uint16_t* out, size_t n_elems) {
    GUARD(ctx);
    const dllm_config& c = ctx->cfg;
    const Layout& L = ctx->L;
    const int d = c.d_model, F = c.ffn, qd = L.qd;
    if (!out) return fail(ctx, DLLM_EINVAL, "null output");
    int rc = DLLM_OK;
    if (layer < 0) {
        if (n_elems < static_cast<size_t>(c.vocab) * d) return fail(ctx, DLLM_EINVAL, "buffer too small");
        if (which == 1) {  // the embedding is row-major
            CK(cudaMemcpyAsync(out, ctx->emb, static_cast<size_t>(c.vocab) * d * 2, cudaMemcpyDeviceToHost,
                               ctx->stream));
            return sync_check(ctx);
        }
        if (which != 2) return fail(ctx, DLLM_EINVAL, "bad tensor");
    } else if (layer >= c.n_layers || which < 0 || which > 6) {
        return fail(ctx, DLLM_EINVAL, "bad tensor");
    }
    // a projection: copy its tile-major matrix, then gather the logical rows
    const int rows = layer < 0 ? c.vocab : (which == 0) ? qd : (which <= 2) ? L.kvd : (which == 3 || which == 6) ? d : F;
    const int cols = layer < 0 ? d : (which == 3) ? qd : (which == 6) ? F : d;
    if (n_elems < static_cast<size_t>(rows) * cols) return fail(ctx, DLLM_EINVAL, "buffer too small");
    const uint8_t* src;
    int phys_rows;
    const size_t unit = L.q4 ? 1 : 2;
    if (layer < 0) {
        src = ctx->head;
        phys_rows = L.head_rows;
    } else {
        src = ctx->wl[layer] + unit * (which <= 2 ? L.w_qkv : which == 3 ? L.w_o : which == 6 ? L.w_d : L.w_gu);
        phys_rows = which <= 2 ? L.qkv_rows : which == 3 ? L.o_rows : which == 6 ? L.d_rows : L.gu_rows;
    }
    const int kb = (cols + 63) / 64;
    const size_t bytes = L.q4 ? static_cast<size_t>(phys_rows / 128) * kb * kQ4TileBytes
                              : static_cast<size_t>(phys_rows) * kb * 64 * 2;
    std::vector<uint8_t> phys(bytes);
    CK(cudaMemcpyAsync(phys.data(), src, bytes, cudaMemcpyDeviceToHost, ctx->stream));
    rc = sync_check(ctx);
    if (rc) return rc;
    // element (physical row pr, column col) as bf16 bits; 4-bit tiles: bf16(d * (q - 8)), the
    // product exact in fp32 and rounded once to nearest even, as the kernel's expansion does
    auto element = [&](int pr, int col) -> uint16_t {
        if (!L.q4) return reinterpret_cast<const uint16_t*>(phys.data())[tiled_index(pr, col, kb)];
        const uint8_t* tile = phys.data() + (static_cast<size_t>(pr >> 7) * kb + (col >> 6)) * kQ4TileBytes;
        const int rr = pr & 127, cc = col & 63;
        uint32_t word;
        memcpy(&word, tile + ((cc >> 3) * 128 + rr) * 4, 4);
        const int q = static_cast<int>((word >> q4_code_shift(cc & 7)) & 15u);
        uint16_t sb;
        memcpy(&sb, tile + 4096 + ((cc >> 5) * 128 + rr) * 2, 2);
        uint32_t sbits = static_cast<uint32_t>(sb) << 16;
        float dsc;
        memcpy(&dsc, &sbits, 4);
        const float w = dsc * static_cast<float>(q - 8);
        uint32_t b;
        memcpy(&b, &w, 4);
        b += 0x7FFFu + ((b >> 16) & 1u);  // round to nearest, ties to even (finite values)
        return static_cast<uint16_t>(b >> 16);
    };
    const int hd = c.head_dim, half = hd / 2;
    for (int r = 0; r < rows; ++r) {
        int pr = r;
        if (layer >= 0 && which <= 2) {  // q/k/v rows are interleaved inside each head
            const int hh = r / hd, i = r % hd;
            pr = (which == 0 ? 0 : qd + (which - 1) * L.kvd) + hh * hd + 2 * (i % half) + i / half;
        } else if (layer >= 0 && (which == 4 || which == 5)) {  // gate/up rows alternate in each tile
            pr = (r / 64) * 128 + 2 * (r % 64) + (which == 5 ? 1 : 0);
        }
        uint16_t* o = out + static_cast<size_t>(r) * cols;
        for (int col = 0; col < cols; ++col) o[col] = element(pr, col);
    }
    return DLLM_OK;
}

int dllm_get_kv(dllm_ctx* ctx, int layer, int which, int seq, int p0, int n, float* out) {
    GUARD(ctx);
    const dllm_config& c = ctx->cfg;
    if (!out || layer < 0 || layer >= c.n_layers || which < 0 || which > 1 || seq < 0 || seq >= c.max_batch || p0 < 0 ||
        n < 0 || p0 + n > c.max_ctx)
        return fail(ctx, DLLM_EINVAL, "bad KV slice");
    const int H = ctx->L.Hkv, hd = c.head_dim, qd = H * hd;  // the cache's K/V heads
    std::vector<uint16_t> buf(static_cast<size_t>(H) * n * hd);
    const __nv_bfloat16* base = ctx->kv + static_cast<size_t>(2 * layer + which) * ctx->L.kv_half;
    for (int h = 0; h < H; ++h)
        CK(cudaMemcpyAsync(buf.data() + static_cast<size_t>(h) * n * hd,
                           base + ((static_cast<size_t>(seq) * H + h) * c.max_ctx + p0) * hd,
                           static_cast<size_t>(n) * hd * 2, cudaMemcpyDeviceToHost, ctx->stream));
    int rc = sync_check(ctx);
    if (rc) return rc;
    for (int p = 0; p < n; ++p)
        for (int h = 0; h < H; ++h)
            for (int i = 0; i < hd; ++i) {
                uint32_t bits = static_cast<uint32_t>(buf[(static_cast<size_t>(h) * n + p) * hd + i]) << 16;
                float f;
                memcpy(&f, &bits, 4);
                out[static_cast<size_t>(p) * qd + h * hd + i] = f;
            }
    return DLLM_OK;
}

}  // extern "C"
