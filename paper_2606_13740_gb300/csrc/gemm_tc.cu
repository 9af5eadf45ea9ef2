// Weight-streaming projections on the 5th-generation tensor cores (tcgen05 + TMEM).
//
// D[m][n] = sum_k W[m][k] * X[n][k]: W are the layer weights (bf16, K-major,
// rows padded to 128), X the activations of the window's tokens (bf16,
// K-major).  The weight rows sit on the UMMA M axis (128 per tile) and the
// tokens on the N axis, so at batch 1 (32 tokens) one UMMA instruction
// covers the whole token set and the kernel is a pure stream of weight
// bytes; at batch 16 (1024 tokens) the same kernel runs 128 x 256 tiles.
//
// One kernel, k_chain, runs one or several projections ("phases") in one
// persistent launch with one CTA per SM: a layer's output projection,
// gate/up, down and the next layer's QKV stream their weights through one
// shared-memory ring, the operand of each phase being loaded once the tiles
// of the previous phase that write it have published completion flags.  A
// single projection (dllm_op_gemm, the first layer's QKV) is a chain of one.
//
// Work in a phase is split "stream-K" style: the flattened (tile, 64-wide
// k-block) iteration space (tiles token-tile-major: the m-tiles of token tile
// 0, then of token tile 1, ..., so that with several token tiles the CTAs
// that read the same weight tile for different token tiles run about in step
// and share it through L2) is cut into one contiguous range per CTA, so
// every SM streams the same number of weight bytes whatever the tile count.
// A tile cut between CTAs is finished by the CTA holding its first k-blocks,
// which are the end of that CTA's range: the other parts store fp32 partials
// and publish each on its own flag, and the finishing CTA polls every part's
// flag at once (bounded), bulk-copies each part's slice into shared memory as
// soon as it is published and adds them to its own accumulator in part order
// (deterministic).  Every CTA waits only on CTAs that wait on nothing later
// than it, and the grid never exceeds the SM count, so all are resident.
// The weights (the context's, stored tile-major) arrive as one contiguous
// bulk copy per 16 KB tile; row-major weights of the single-projection entry
// points arrive through a 2-D tensor map.
//
// Epilogues are fused: residual add with the next RMSNorm's statistics,
// RoPE + KV-cache write, SwiGLU, and the LM head's per-tile softmax
// statistics; the consumers of a residual apply RMSNorm as a per-token scale
// of their fp32 accumulators.  The epilogue runs once per tile on the step's
// critical path, so it avoids dependent chains of global loads (everything
// it reads is loaded before it stores, or staged early) and keeps its code
// compact.
#include "common.cuh"
#include "internal.h"

#include <climits>

namespace dllm {

constexpr int kBM = 128;    // UMMA M
constexpr int kBK = 64;     // K elements per stage: one 128-byte swizzle row
constexpr uint32_t kABytes = kBM * kBK * 2;
constexpr int kFullSmem = 227 * 1024;
static int g_stream_budget = kChainSmemShared;  // single projections: shared-memory plan
constexpr int kTicketStride = 32;  // a tile's part flags: one 128-byte line (parts 1..31)
constexpr int kEpiGroup = 16;      // epilogue columns processed side by side: half a 32-token chunk
constexpr int kEpiWarps = 8;       // two per TMEM lane quarter, one per half chunk
constexpr int kEpiThreads = kEpiWarps * 32;

// Timeline trace slots per CTA (when EpiArgs::trace is set).
enum { kTrStart = 0, kTrPrologue = 1, kTrFirstData = 2, kTrLastData = 3, kTrEpiDone = 4, kTrExit = 5, kTrSm = 6,
       kTrDepWait = 7, kTrAccReady = 8, kTrPartStored = 9, kTrTicket = 10, kTrReduced = 11, kTrIsLast = 12,
       kTrTile = 13, kTrEpiPass1 = 14, kTrPublished = 15, kTrSlots = 16 };

__device__ __forceinline__ unsigned smid() {
    unsigned id;
    asm volatile("mov.u32 %0, %%smid;" : "=r"(id));
    return id;
}

__device__ __forceinline__ int owner_of(long long i, long long total, int G) {
    return static_cast<int>(((i + 1) * G + total - 1) / total) - 1;
}

__device__ __forceinline__ long long range_begin(int c, long long total, int G) { return total * c / G; }


struct EpiSmem {
    float* rs;    // [256] per-column RMSNorm scale of the current token tile
    float* red;   // [4][256] cross-warp / quarter partial sums
    int* kvs;     // [256] per-sequence first window position (QKV); current ids of the token tile (LM head)
    float* theta; // [128] rotation frequency of each tile row's feature pair (QKV)
    uint8_t* stg;  // staging of a 32-token chunk's bf16 outputs, 8 KB (for tiles of more than one chunk its
                   // own memory: the next chunk's partial slices arrive meanwhile)
    const int* rows;  // the launch's device-resolved row count (-1: the plans as given)
};

// The plan of a phase in a launch whose rows are resolved on the device (rows >= 0): only the
// token tiles that hold rows [0, rows), their iterations split anew over the CTAs (a phase with
// no rows gets grid 0: every role skips it).
__device__ __forceinline__ GemmPlan phase_plan(const ChainPhase& P, int rows) {
    GemmPlan p = P.p;
    if (rows >= 0) {
        const int nt = min(p.n_tiles, (rows + p.ntile - 1) / p.ntile);
        p.n_tiles = nt;
        p.total = static_cast<long long>(p.m_tiles) * nt * p.kb;
        const long long min_iters = (p.kb + 29) / 30;  // at most 31 parts per tile, as on the host
        if (p.grid > p.total / min_iters) p.grid = static_cast<int>(p.total / min_iters);
    }
    return p;
}

// RMSNorm scale of every column of token tile nt: rs[c] = rsqrt(sum_t sq[t][col] / dim + eps).
// The epilogue threads, 4 per column (each over a quarter of the statistics, loads
// independent), summed in a fixed order: deterministic.
__device__ __forceinline__ void compute_norm_scale(const EpiArgs& ep, const GemmPlan& p, int nt, const EpiSmem& sm,
                                                   int e) {
    for (int item = e; item < 4 * p.ntile; item += kEpiThreads) {
        const int c = item % p.ntile, q = item / p.ntile;
        const int col = nt * p.ntile + c;
        float s = 0.0f;
        if (col < p.N) {
            float a[8];
            int t = q;
            for (; t + 28 < ep.n_sq; t += 32) {
#pragma unroll
                for (int u = 0; u < 8; ++u) a[u] = ep.sq_in[static_cast<size_t>(t + 4 * u) * p.N + col];
#pragma unroll
                for (int u = 0; u < 8; ++u) s += a[u];
            }
            for (; t < ep.n_sq; t += 4) s += ep.sq_in[static_cast<size_t>(t) * p.N + col];
        }
        sm.red[q * 256 + c] = s;
    }
    named_bar(1, kEpiThreads);
    for (int c = e; c < p.ntile; c += kEpiThreads) {
        const float s = ((sm.red[c] + sm.red[256 + c]) + sm.red[512 + c]) + sm.red[768 + c];
        sm.rs[c] = rsqrtf(s / static_cast<float>(ep.norm_dim) + ep.eps);
    }
    named_bar(1, kEpiThreads);
}

// (cos, sin) of an angle: one out-of-line copy, called twice per chunk on the common path.
__device__ __noinline__ float2 rot_cs(float angle) {
    float sn, cn;
    sincosf(angle, &sn, &cn);
    return make_float2(cn, sn);
}

// ------------------------------------------------------------------ epilogues
// Sum of v[0..N-1] (N a power of two <= 32) over the 32 lanes of a warp, scattered:
// afterwards the 32/N lanes c*(32/N) .. c*(32/N)+32/N-1 hold the total of column c in v[0].
// N-1 + log2(32/N) shuffles in a fixed order.
template <int N>
__device__ __forceinline__ void warp_reduce_scatter(float* v, int lane) {
#pragma unroll
    for (int w = 16, h = N / 2; h >= 1; w >>= 1, h >>= 1) {
        const bool upper = (lane & w) != 0;
#pragma unroll
        for (int i = 0; i < h; ++i) {
            const float send = upper ? v[i] : v[i + h];
            const float keep = upper ? v[i + h] : v[i];
            v[i] = keep + __shfl_xor_sync(0xffffffffu, send, w);
        }
    }
#pragma unroll
    for (int w = 16 / N; w >= 1; w >>= 1) v[0] += __shfl_xor_sync(0xffffffffu, v[0], w);
}

// What a QKV epilogue thread needs besides the accumulator, from the tile and chunk alone: its
// row's part (q, K or V) and position in the head, the rotation at its first column and the
// per-column step (angle addition along the positions, when all 32 columns are consecutive
// positions of one sequence's window), and the 32-byte store it makes after the staging (token
// t/8, tile features 16 (t%8) .. +15: part of one head's run at the token's row of the q
// tensor, the K/V cache or, for tracked prefix rows, the side buffers).  A finisher that waits
// for other parts of its tile builds it before the wait.
struct QkvPlan {
    int part, pp, fi, bl;
    bool run;
    float cn, sn, cd, sd, theta;
    uint4* dst;  // null: no store
    bool bad;    // a window position outside the cache
};
__device__ __forceinline__ QkvPlan qkv_plan(const EpiArgs& ep, const GemmPlan& p, int mt, int col0, int rt,
                                            const EpiSmem& sm, int e, int half) {
    QkvPlan q;
    const int row = mt * kBM + rt;
    // q rows [0, qd), k rows [qd, qd + kvd), v rows [qd + kvd, qd + 2 kvd): the same part for
    // the whole tile (qd and kvd are multiples of 128)
    const int qd = ep.H * ep.hd;
    q.part = row < qd ? 0 : (row < ep.v_row0 ? 1 : 2);
    const int f = row - (q.part == 0 ? 0 : (q.part == 1 ? qd : ep.v_row0));
    q.pp = f % ep.hd;
    q.fi = (q.pp >> 1) + (q.pp & 1) * (ep.hd >> 1);
    q.theta = sm.theta[rt];
    q.bl = col0 / ep.T;
    q.run = min(col0 + 31, p.N - 1) / ep.T == q.bl && min(col0 + 31, p.N - 1) - q.bl * ep.T < ep.Tw;
    q.cn = 1.0f;
    q.sn = 0.0f;
    q.cd = 1.0f;
    q.sd = 0.0f;
    if (q.part < 2 && q.run) {
        const float2 a = rot_cs(static_cast<float>(sm.kvs[q.bl] + (col0 + kEpiGroup * half - q.bl * ep.T)) * q.theta);
        const float2 d = rot_cs(q.theta);
        q.cn = a.x;
        q.sn = a.y;
        q.cd = d.x;
        q.sd = d.y;
    }
    const int tok = e >> 3, f0 = (e & 7) * 16;
    const int col = col0 + tok;
    q.dst = nullptr;
    q.bad = false;
    if (col < p.N) {
        const int b = min(col / ep.T, ep.n_seq - 1);
        const int ts = col - b * ep.T;
        const bool tracked = ts >= ep.Tw;  // sparse cache refresh: K/V to the side buffers
        const int pos = tracked ? ep.trk[b * ep.R + ts - ep.Tw] : sm.kvs[b] + ts;
        const int base = q.part == 0 ? 0 : (q.part == 1 ? qd : ep.v_row0);  // the part's first row
        const int head = (mt * kBM - base + f0) / ep.hd;
        const int heads = q.part == 0 ? ep.H : ep.Hkv;  // q: query heads; K/V: the cache's heads
        const int fi0 = f0 % ep.hd;
        if (tracked && q.part > 0) {
            if (pos >= 0) {
                __nv_bfloat16* side = q.part == 1 ? ep.kside : ep.vside;
                q.dst = reinterpret_cast<uint4*>(
                    side + ((static_cast<size_t>(b) * heads + head) * ep.R + (ts - ep.Tw)) * ep.hd + fi0);
            }
        } else if (tracked || (pos >= 0 && pos < ep.cap)) {
            const size_t plane = q.part == 0 ? static_cast<size_t>(ep.T) : static_cast<size_t>(ep.cap);
            const size_t r = (static_cast<size_t>(b) * heads + head) * plane + (q.part == 0 ? ts : pos);
            __nv_bfloat16* base_ptr = q.part == 0 ? ep.q : (q.part == 1 ? ep.kc : ep.vc);
            q.dst = reinterpret_cast<uint4*>(base_ptr + r * ep.hd + fi0);
        } else {
            q.bad = true;
        }
    }
    return q;
}

// Epilogue of a 32-token chunk, compact: each epilogue thread takes its TMEM lane (tile row)
// and one half of the chunk, 16 columns read from TMEM (t_src; for the residual, the old x of
// a narrow tile was staged at t_x before the accumulator was ready), so its code stays small
// and no global load waits on a store.  The 16 columns run side by side with no branch between
// them (stores are predicated), so their dependent chains (shuffles, special functions)
// overlap; the chunk's outputs are staged in shared memory and stored in 16-byte pieces.
// Residual epilogue in two passes (PASS 1: the bf16 copy, the next projection's operand, and
// the RMSNorm partial sums; PASS 2: the fp32 residual and the sums' store), so the tile can be
// published to the next phase's operand producer between them; PASS 0: both at once.
template <int EPI, int PASS = 0>
__device__ __forceinline__ void epilogue_c32(const EpiArgs& ep, const GemmPlan& p, int mt, int col0, int c_in,
                                             int rt, uint32_t t_src, uint32_t t_x, const EpiSmem& sm,
                                             int e, int half, int quarter, int lane, int* status,
                                             const float* a_in = nullptr, const QkvPlan* qkv_pre = nullptr,
                                             const float* x_in = nullptr) {
    // col0: the chunk's first token column; c_in: its offset inside the token tile (index into
    // the tile's RMSNorm scales and staged ids).  The thread's 16 accumulator columns come from
    // a_in (a finisher's sum of the parts, in registers), else from TMEM at t_src.  The old
    // residual (pass 1) comes from TMEM (t_x), else from global memory (a warp's 32 rows of a
    // token are one 128-byte line; L2 only: other CTAs wrote them in earlier phases); pass 1
    // leaves the new residual in the accumulator, where pass 2 reads it.  e: the epilogue thread (0 .. kEpiThreads-1), half: which 16 columns of the
    // chunk.  qkv_pre: the QKV plan, built ahead (null: built here).
    constexpr int GW = kEpiGroup;  // columns per group
    constexpr int LS = 32 / GW;    // lanes sharing one column's sum after the scatter
    const int row = mt * kBM + rt;
    const bool scale = (EPI == EPI_QKV || EPI == EPI_SWIGLU || EPI == EPI_LMHEAD) && ep.sq_in != nullptr;
    QkvPlan qp;
    if constexpr (EPI == EPI_QKV) qp = qkv_pre ? *qkv_pre : qkv_plan(ep, p, mt, col0, rt, sm, e, half);
    // QKV state: feature, rotation (angle-addition recurrence along the positions)
    int part = 0, pp = 0, fi = 0, bl = 0;
    bool run = true;
    float cn = 1.0f, sn = 0.0f, cd = 1.0f, sd = 0.0f, theta = 0.0f;
    if constexpr (EPI == EPI_QKV) {
        part = qp.part;
        pp = qp.pp;
        fi = qp.fi;
        bl = qp.bl;
        run = qp.run;
        cn = qp.cn;
        sn = qp.sn;
        cd = qp.cd;
        sd = qp.sd;
        theta = qp.theta;
    }
    bool lm_ok = false;
    if constexpr (EPI == EPI_LMHEAD) lm_ok = row < ep.V && row != ep.mask_id;
    static_assert(32 / GW == 2, "one column group per half chunk");
    {
        const int g = half;

        const int cg = col0 + GW * g;  // first column of the group
        float a[GW];
        if (a_in) {
#pragma unroll
            for (int u = 0; u < GW; ++u) a[u] = a_in[u];
        } else {
            tmem_ld_32xn<GW>(t_src + static_cast<uint32_t>(GW * g), a);
        }
        if (scale) {
#pragma unroll
            for (int u = 0; u < GW; ++u) a[u] *= sm.rs[c_in + GW * g + u];
        }
        if constexpr (EPI == EPI_F32) {
#pragma unroll
            for (int u = 0; u < GW; ++u)
                if (row < p.M && cg + u < p.N) ep.out[static_cast<size_t>(cg + u) * ep.ld_out + row] = a[u];
        } else if constexpr (EPI == EPI_RESID) {
            float xo[GW], ss[GW];
            if constexpr (PASS == 2) {
#pragma unroll
                for (int u = 0; u < GW; ++u) xo[u] = a[u];
            } else {
                if (t_x) {
                    tmem_ld_32xn<GW>(t_x + static_cast<uint32_t>(GW * g), xo);
                } else if (x_in) {
#pragma unroll
                    for (int u = 0; u < GW; ++u) xo[u] = x_in[u];
                } else {
#pragma unroll
                    for (int u = 0; u < GW; ++u)
                        xo[u] = (row < p.M && cg + u < p.N) ? __ldcg(ep.out + static_cast<size_t>(cg + u) * ep.ld_out + row)
                                                            : 0.0f;
                }
#pragma unroll
                for (int u = 0; u < GW; ++u) xo[u] += a[u];
            }
            if constexpr (PASS == 1) tmem_st_32xn<GW>(t_src + static_cast<uint32_t>(GW * g), xo);
#pragma unroll
            for (int u = 0; u < GW; ++u) {
                const bool ok = row < p.M && cg + u < p.N;
                ss[u] = ok ? xo[u] * xo[u] : 0.0f;
                if constexpr (PASS == 0) {
                    if (ok) {
                        const size_t o = static_cast<size_t>(cg + u) * ep.ld_out + row;
                        ep.out[o] = xo[u];
                        ep.xb[o] = __float2bfloat16_rn(xo[u]);
                    }
                } else if constexpr (PASS == 1) {  // token-major staging, stored below in 16-byte pieces
                    reinterpret_cast<__nv_bfloat16*>(sm.stg)[(GW * g + u) * kBM + rt] = __float2bfloat16_rn(xo[u]);
                } else {  // fp32: a warp's 32 rows of one token are one 128-byte line
                    if (ok) ep.out[static_cast<size_t>(cg + u) * ep.ld_out + row] = xo[u];
                }
            }
            if constexpr (PASS != 2) {
                warp_reduce_scatter<GW>(ss, lane);
                if (lane % LS == 0) sm.red[(c_in / 32) * 128 + quarter * 32 + GW * g + lane / LS] = ss[0];
            }
        } else if constexpr (EPI == EPI_QKV) {
            // positions and rotations of the group's 8 columns first (the rare tile that spans
            // sequences takes the out-of-line sincos per column), then the branch-free column pass
            int bs[GW], ts[GW];
            float cs[GW], ss[GW];
            if (run) {
#pragma unroll
                for (int u = 0; u < GW; ++u) {
                    bs[u] = bl;
                    ts[u] = cg + u - bl * ep.T;
                    cs[u] = cn;
                    ss[u] = sn;
                    const float c2 = cn * cd - sn * sd;  // angle-addition step to the next position
                    sn = sn * cd + cn * sd;
                    cn = c2;
                }
            } else {
#pragma unroll
                for (int u = 0; u < GW; ++u) {
                    const int b = min((cg + u) / ep.T, ep.n_seq - 1);
                    bs[u] = b;
                    ts[u] = cg + u - b * ep.T;
                    // a window row, or (sparse cache refresh) a tracked prefix position
                    const int ps = ts[u] < ep.Tw ? sm.kvs[b] + ts[u] : max(ep.trk[b * ep.R + ts[u] - ep.Tw], 0);
                    const float2 r = rot_cs(static_cast<float>(ps) * theta);
                    cs[u] = r.x;
                    ss[u] = r.y;
                }
            }
            float xp[GW];
#pragma unroll
            for (int u = 0; u < GW; ++u) xp[u] = __shfl_xor_sync(0xffffffffu, a[u], 1);
            // staged token-major in feature order ([32][128]: the tile's head(s) side by side),
            // stored below in 16-byte pieces
            __nv_bfloat16* st = reinterpret_cast<__nv_bfloat16*>(sm.stg) + (rt / ep.hd) * ep.hd + fi;
#pragma unroll
            for (int u = 0; u < GW; ++u) {
                float x = a[u];
                if (part < 2) x = (pp & 1) ? (x * cs[u] + xp[u] * ss[u]) : (x * cs[u] - xp[u] * ss[u]);
                st[(GW * g + u) * kBM] = __float2bfloat16_rn(x);
            }
        } else if constexpr (EPI == EPI_SWIGLU) {
            // tile row 2f is gate feature f, row 2f+1 the matching up row
            const int f = mt * 64 + (rt >> 1);
            const bool gate_lane = (rt & 1) == 0 && f < ep.F;
            float up[GW];
#pragma unroll
            for (int u = 0; u < GW; ++u) up[u] = __shfl_xor_sync(0xffffffffu, a[u], 1);
            // staged token-major ([32][64] features), stored below in 16-byte pieces
            __nv_bfloat16* st = reinterpret_cast<__nv_bfloat16*>(sm.stg) + (rt >> 1);
#pragma unroll
            for (int u = 0; u < GW; ++u) {
                const __nv_bfloat16 hv = __float2bfloat16_rn(__fdividef(a[u], 1.0f + __expf(-a[u])) * up[u]);
                if (gate_lane) st[(GW * g + u) * 64] = hv;
            }
        } else if constexpr (EPI == EPI_LMHEAD) {
            // this warp's (max, argmax, sum exp) over its 32 rows, for the 8 columns side by side
            float m[GW], e[GW];
            int idx[GW];
#pragma unroll
            for (int u = 0; u < GW; ++u) {
                m[u] = lm_ok ? a[u] : -INFINITY;
                idx[u] = lm_ok ? row : INT_MAX;
            }
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) {
#pragma unroll
                for (int u = 0; u < GW; ++u) {
                    const float om = __shfl_xor_sync(0xffffffffu, m[u], off);
                    const int oi = __shfl_xor_sync(0xffffffffu, idx[u], off);
                    const bool take = om > m[u] || (om == m[u] && oi < idx[u]);
                    m[u] = take ? om : m[u];
                    idx[u] = take ? oi : idx[u];
                }
            }
#pragma unroll
            for (int u = 0; u < GW; ++u) e[u] = (lm_ok && m[u] != -INFINITY) ? __expf(a[u] - m[u]) : 0.0f;
            if (lane == 0) {
#pragma unroll
                for (int u = 0; u < GW; ++u) {
                    sm.red[(quarter * 32 + GW * g + u) * 3] = m[u];
                    sm.red[(quarter * 32 + GW * g + u) * 3 + 2] = __int_as_float(idx[u]);
                }
            }
            warp_reduce_scatter<GW>(e, lane);
            if (lane % LS == 0) sm.red[(quarter * 32 + GW * g + lane / LS) * 3 + 1] = e[0];
#pragma unroll
            for (int u = 0; u < GW; ++u) {
                const int col = cg + u;
                if (ep.logits && row < ep.V && col < p.N) ep.logits[static_cast<size_t>(col) * ep.V + row] = a[u];
                if (col < p.N && row == sm.kvs[c_in + GW * g + u]) ep.zcur[col] = a[u];  // current ids staged
            }
        }
    }
    if constexpr (EPI == EPI_QKV) {
        // thread t stores token t/8, tile features 16 (t%8) .. +15 (the plan's destination)
        named_bar(1, kEpiThreads);
        if (qp.dst) {
            const int t = e, tok = t >> 3, f0 = (t & 7) * 16;
            const uint4* src =
                reinterpret_cast<const uint4*>(reinterpret_cast<const __nv_bfloat16*>(sm.stg) + tok * kBM + f0);
#pragma unroll
            for (int i = 0; i < 2; ++i) qp.dst[i] = src[i];
        }
        if (qp.bad) atomicOr(status, kStatusBadIndex);
        named_bar(1, kEpiThreads);  // the staging memory is free again
    } else if constexpr (EPI == EPI_SWIGLU) {
        // thread t stores token t/8, features 8 (t%8) .. +7 of the tile's 64
        named_bar(1, kEpiThreads);
        const int t = e, tok = t >> 3, f0 = (t & 7) * 8;
        const int col = col0 + tok;
        if (col < p.N) {
            const uint4* src =
                reinterpret_cast<const uint4*>(reinterpret_cast<const __nv_bfloat16*>(sm.stg) + tok * 64 + f0);
            const int fg = mt * 64 + f0;  // F is a multiple of 8: each 8-feature piece is all in or all out
            if (fg < ep.F) *reinterpret_cast<uint4*>(ep.h + static_cast<size_t>(col) * ep.F + fg) = *src;
        }
        named_bar(1, kEpiThreads);
    }
    if constexpr (EPI == EPI_RESID && PASS == 1) {
        // the staged chunk: thread t stores token t/8, features 16 (t%8) .. +15 of the tile
        named_bar(1, kEpiThreads);
        const int t = e, tok = t >> 3, f0 = (t & 7) * 16;
        const int col = col0 + tok;
        if (col < p.N) {
            const uint4* src =
                reinterpret_cast<const uint4*>(reinterpret_cast<const __nv_bfloat16*>(sm.stg) + tok * kBM + f0);
            uint4* dst = reinterpret_cast<uint4*>(ep.xb + static_cast<size_t>(col) * ep.ld_out + mt * kBM + f0);
#pragma unroll
            for (int i = 0; i < 2; ++i) dst[i] = src[i];
        }
        named_bar(1, kEpiThreads);  // the staging memory is free again
    }
    if constexpr (EPI == EPI_RESID && PASS == 0) {
        named_bar(1, kEpiThreads);
        if (e < 32) {
            const int col = col0 + lane;
            const float* rd = sm.red + (c_in / 32) * 128;
            if (col < p.N)
                ep.sq_out[static_cast<size_t>(mt) * p.N + col] = ((rd[lane] + rd[32 + lane]) + rd[64 + lane]) + rd[96 + lane];
        }
        named_bar(1, kEpiThreads);
    } else if constexpr (EPI == EPI_RESID && PASS == 2) {
        // the chunk's four quarter sums, written by its first pass (the barriers since then order
        // them; the next writer of these words comes after the tile's next barrier)
        if (e < 32) {
            const int col = col0 + lane;
            const float* rd = sm.red + (c_in / 32) * 128;
            if (col < p.N)
                ep.sq_out[static_cast<size_t>(mt) * p.N + col] = ((rd[lane] + rd[32 + lane]) + rd[64 + lane]) + rd[96 + lane];
        }
    } else if constexpr (EPI == EPI_LMHEAD) {
        named_bar(1, kEpiThreads);
        if (e < 32) {  // merge the four row quarters in a fixed order
            const int col = col0 + lane;
            float m = -INFINITY, s = 0.0f;
            int idx = INT_MAX;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float* r = sm.red + (q * 32 + lane) * 3;
                const float m2 = r[0], s2 = r[1];
                const int i2 = __float_as_int(r[2]);
                if (m2 == -INFINITY) continue;
                if (m == -INFINITY) {
                    m = m2;
                    s = s2;
                    idx = i2;
                } else if (m2 > m) {
                    s = s * __expf(m - m2) + s2;
                    m = m2;
                    idx = i2;
                } else if (m2 == m) {
                    s += s2;
                    idx = min(idx, i2);
                } else {
                    s += s2 * __expf(m2 - m);
                }
            }
            if (col < p.N) {
                float* o = ep.lm_part + (static_cast<size_t>(col) * p.m_tiles + mt) * 3;
                o[0] = m;
                o[1] = s;
                o[2] = __int_as_float(idx);
            }
        }
        named_bar(1, kEpiThreads);
    }
}

// ================================================================== chained projections
// k_chain runs the phases of a ChainArgs in one launch, one CTA per SM.  Roles (352
// threads): warp 0 = weight producer (never waits on data: weights are constant, so it runs
// ahead by the whole ring, across phase boundaries), warp 6 = operand producer (waits for
// the completion flag of the tile that writes each X k-block), warp 1 = TMEM owner and MMA
// issuer, warps 2..5 and 7..10 = epilogue (two warps per TMEM lane quarter).  The operand
// producer's and the MMA issuer's loops run warp-wide, one elected lane issuing.  Ring stages,
// TMEM accumulators and their barriers are shared by all phases; a running iteration counter
// gives every stage its use parity.
constexpr int kChainThreads = 64 + 32 + 32 * kEpiWarps;
// 4-bit weights: warps 11..14 expand the raw tiles into the bf16 A stages
constexpr int kDeqWarp0 = 11, kDeqWarps = 4;
constexpr int kChainThreadsQ4 = kChainThreads + 32 * kDeqWarps;
constexpr int kMaxDepTiles = 1024;  // the operand producer keeps a readiness bit per producing tile: 32 per lane

struct ChainEpiState {
    int acc;
    uint32_t acc_phase;
    uint32_t red_phase;
};

__device__ __forceinline__ int chain_tag(const ChainArgs& ca) {
    return ca.epoch ? *reinterpret_cast<const volatile int*>(ca.epoch) * ca.tag_mul + ca.tag_add : ca.tag_add;
}

// Wait (bounded) until flag == tag.  Returns false after raising *abort on a timeout.
__device__ __forceinline__ bool wait_flag(const int* flag, int tag, volatile int* abort, int* status) {
    if (ld_acquire(flag) == tag) return true;
    const long long t0 = spin_clock();
    while (ld_acquire(flag) != tag) {
        if (*abort) return false;
        if (spin_clock() - t0 > kWaitLimitCycles) {
            *abort = 1;
            atomicOr(status, kStatusTimeout);
            return false;
        }
    }
    return true;
}

// A finisher's wait for parts q0 .. q0+qn-1 of its tile (flag q == tag): warp ew 0 polls them,
// lane q reading flag q, so one round trip covers the group; then every epilogue thread passes
// a barrier.  False when the launch is unwinding (a stalled wait sets the abort flag and the
// status word).
__device__ __forceinline__ bool wait_parts(const int* flags, int q0, int qn, int tag, int ew, int lane,
                                           volatile int* s_abort, int* status) {
    if (ew == 0) {
        const long long t0 = spin_clock();
        for (;;) {
            const bool ok = lane < q0 || lane >= q0 + qn || ld_acquire(flags + lane) == tag;
            if (__all_sync(0xffffffffu, ok)) break;
            int give_up = 0;
            if (lane == 0) give_up = (*s_abort || spin_clock() - t0 > kWaitLimitCycles) ? 1 : 0;
            if (__shfl_sync(0xffffffffu, give_up, 0)) {  // warp-uniform decision
                if (lane == 0 && !*s_abort) {
                    *s_abort = 1;
                    atomicOr(status, kStatusTimeout);
                }
                break;
            }
            __nanosleep(32);
        }
    }
    return !named_bar_any(1, kEpiThreads, *s_abort != 0);
}

// The epilogue warps' share of one phase: every tile of this CTA's range.
// WIDE: token tiles of several 32-token chunks (split tiles reduced through the staging
// slots); else one chunk (split tiles reduced in registers): each its own code.
template <int EPI, int DP, bool WIDE>
__device__ __forceinline__ void chain_phase_epilogue(const ChainArgs& ca, int ph, int tag, uint8_t* red_stage,
                                                  uint64_t* tfull, uint64_t* tempty, uint64_t* redbar,
                                                  volatile int* s_abort, uint32_t tmem_base, const EpiSmem& esm,
                                                  ChainEpiState& es) {
    const ChainPhase& P = ca.ph[ph];
    const GemmPlan p = phase_plan(P, *esm.rows);
    const EpiArgs& ep = P.ep;
    int* status = ca.status;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int ew = warp < 6 ? warp - 2 : warp - 3;  // epilogue warps 2..5 and 7..10
    const int e = ew * 32 + lane;                     // epilogue thread
    const int half = ew >> 2;                         // columns 16 half .. +15 of every chunk
    const int quarter = warp & 3;                     // TMEM lane quarter = tile rows 32 quarter ..
    const int rt = quarter * 32 + lane;
    const int G = p.grid;
    if (static_cast<int>(blockIdx.x) >= G) return;
    const long long it0 = range_begin(blockIdx.x, p.total, G);
    const long long it1 = range_begin(blockIdx.x + 1, p.total, G);
    if (it0 >= it1) return;
    unsigned long long* tr = ep.trace ? ep.trace + static_cast<size_t>(blockIdx.x) * kTrSlots : nullptr;
    if (tr && threadIdx.x == 64) {
        tr[kTrSm] = smid();
        for (int i = kTrAccReady; i < kTrSlots; ++i) tr[i] = 0;
    }
    // every tile of the previous phase: its RMSNorm statistics and residual rows are read here
    if (ph > 0 && ca.ph[ph - 1].done) {
        const ChainPhase& Q = ca.ph[ph - 1];
        const int* qdone = Q.done2 ? Q.done2 : Q.done;  // the residual phases finish their tiles in two steps
        if (ew == 0) {
            const int n = Q.p.m_tiles * Q.p.n_tiles;
            for (int i = lane; i < n; i += 32)
                if (!wait_flag(qdone + i, tag, s_abort, status)) break;
        }
        if (named_bar_any(1, kEpiThreads, *s_abort != 0)) return;
    }
    if (tr && threadIdx.x == 64) tr[kTrDepWait] = global_ns();
    if constexpr (EPI == EPI_QKV) {
        for (int b = e; b < ep.n_seq; b += kEpiThreads) esm.kvs[b] = ep.seq_kv[b];
        if (half == 0) esm.theta[rt] = ep.theta[(rt % ep.hd) >> 1];
        named_bar(1, kEpiThreads);
    }
    const int nchunks = p.ntile / 32;
    constexpr int kPass1 = EPI == EPI_RESID ? 1 : 0;  // the residual epilogue runs in two passes
    const size_t slot_floats = static_cast<size_t>(p.ntile) * kBM;
    // TMEM: two accumulators of acc_cols columns, then (token tiles up to 128) the staged old
    // residual of the finisher's tile, x_cols columns
    const uint32_t t_x =
        ca.x_cols ? tmem_base + static_cast<uint32_t>(2 * ca.acc_cols) + (static_cast<uint32_t>(quarter * 32) << 16)
                  : 0u;
    int rs_nt = -1, ids_nt = -1;
    long long prepared = -1;
    float v[16];
    // Work a finisher needs before its accumulator: the RMSNorm scale of its token tile, the
    // LM head's current ids of the token tile, and (residual, 32-token tiles) the old x staged
    // in TMEM.  Done as early as possible: for a contributor tile, ahead of it for the finisher
    // tile that follows in the range.
    auto prepare = [&](long long ptile) {
        if (ptile == prepared) return;
        prepared = ptile;
        const int pnt = static_cast<int>(ptile / p.m_tiles);
        const int pmt = static_cast<int>(ptile - static_cast<long long>(pnt) * p.m_tiles);
        if constexpr (EPI == EPI_QKV || EPI == EPI_SWIGLU || EPI == EPI_LMHEAD) {
            if (ep.sq_in && pnt != rs_nt) {
                compute_norm_scale(ep, p, pnt, esm, e);
                rs_nt = pnt;
            }
        }
        if constexpr (EPI == EPI_LMHEAD) {
            if (pnt != ids_nt) {
                for (int c = e; c < p.ntile; c += kEpiThreads) {
                    const int col = pnt * p.ntile + c;
                    esm.kvs[c] = col < p.N ? ep.cur_tok[col] : -1;
                }
                named_bar(1, kEpiThreads);
                ids_nt = pnt;
            }
        }
        if constexpr (EPI == EPI_RESID) {
            if (t_x) {
                const int row = pmt * kBM + rt;
                for (int c = 0; c < nchunks; ++c) {
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const int col = pnt * p.ntile + c * 32 + half * 16 + j;
                        v[j] = (row < p.M && col < p.N) ? ep.out[static_cast<size_t>(col) * ep.ld_out + row] : 0.0f;
                    }
                    tmem_st_32x16(t_x + static_cast<uint32_t>(c * 32 + half * 16), v);
                }
            }
        }
    };
    for (long long it = it0; it < it1;) {
        const long long tile = it / p.kb;
        const int k_lo = static_cast<int>(it - tile * p.kb);
        const long long tend = (tile + 1) * p.kb;
        const int k_hi = static_cast<int>((it1 < tend ? it1 : tend) - tile * p.kb);
        const int nt = static_cast<int>(tile / p.m_tiles);
        const int mt = static_cast<int>(tile - static_cast<long long>(nt) * p.m_tiles);
        const bool whole = (k_lo == 0 && k_hi == p.kb);
        int c_first = 0, c_last = 0;
        bool reducer = false;
        if (!whole) {
            c_first = owner_of(tile * p.kb, p.total, G);
            c_last = owner_of(tile * p.kb + p.kb - 1, p.total, G);
            reducer = static_cast<int>(blockIdx.x) == c_first;
        }
        const bool finisher = whole || reducer;
        // a contributor's range goes on into a tile whose first k-blocks it holds: a finisher
        if (finisher) prepare(tile);
        else if (tend < it1) prepare(tile + 1);
        // the accumulator (a one-chunk split tile's finisher waits for it after fetching its
        // second part, below)
        const bool late_acc = reducer && !WIDE;
        if (!late_acc) {
            mbar_wait(&tfull[es.acc], es.acc_phase, s_abort, status);
            if (named_bar_any(1, kEpiThreads, *s_abort != 0)) {
                cp_async_wait<0>();  // no copy lands in shared memory after the launch has ended
                return;
            }
            if (tr && threadIdx.x == 64) {
                tr[kTrAccReady] = global_ns();
                tr[kTrTile] = static_cast<unsigned long long>(tile);
            }
            tc_fence_after();
        }
        const uint32_t t_acc = tmem_base + static_cast<uint32_t>(es.acc * ca.acc_cols) +
                               (static_cast<uint32_t>(quarter * 32) << 16);
        if (whole) {
            // the compact epilogue per 32-column chunk, straight from the accumulator in TMEM
            for (int c = 0; c < nchunks; ++c) {
                epilogue_c32<EPI, kPass1>(ep, p, mt, nt * p.ntile + c * 32, c * 32, rt,
                                          t_acc + static_cast<uint32_t>(c * 32),
                                          t_x ? t_x + static_cast<uint32_t>(c * 32) : 0u, esm, e, half, quarter, lane,
                                          status);
            }
        } else if (!reducer) {
            float* my_part = P.partials + static_cast<size_t>(blockIdx.x) * slot_floats;
            for (int c = 0; c < nchunks; ++c) {
                tmem_ld_32x16(t_acc + static_cast<uint32_t>(c * 32 + half * 16), v);
                float4* dst = reinterpret_cast<float4*>(my_part);
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    dst[static_cast<size_t>(c * 8 + half * 4 + j) * kBM + rt] =
                        make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
            }
            // the partial is in registers' way out: the accumulator is free again
            tc_fence_before();
            mbar_arrive(&tempty[es.acc]);
            named_bar(1, kEpiThreads);
            if (threadIdx.x == 64) {  // part q of the tile publishes its partial on flag q
                if (tr) tr[kTrPartStored] = global_ns();
                st_release(&P.tickets[tile * kTicketStride + (static_cast<int>(blockIdx.x) - c_first)], tag);
            }
        }
        if (reducer) {
            // Part q's partial, chunk c (32 columns), is the contiguous 16 KB slice [c*8 + j][row]
            // float4.  The slices go through the nsl staging slots (one or two) in one stream,
            // chunk-major (slice s = chunk s / (nparts-1), part s % (nparts-1) + 1, slot s % nsl):
            // each copy is issued as soon as its part has published (flag q == tag) and its
            // slot's previous slice is added, so a chunk's slices arrive during the previous
            // chunk's epilogue.  The sum runs over q in order, so it does not depend on the arrival
            // order.  (Tiles of one 32-token chunk take the direct path below instead.)
            const int nparts = c_last - c_first + 1;
            const int np1 = nparts - 1;
            const int nslices = nchunks * np1;
            int* flags = &P.tickets[tile * kTicketStride];
            constexpr uint32_t slice_bytes = 32 * kBM * 4;
            const int nsl = ca.red_bytes >= 2 * static_cast<int>(slice_bytes) ? 2 : 1;
            uint32_t ready = 0;     // warp 2: parts seen published (bit q)
            uint32_t inflight = 0;  // thread 64: slots with a copy not yet waited for
            // warp 2, warp-uniform: make sure slice s's part has published, polling every part's
            // flag at once (lane i reads flag i, so one round trip covers them all), then thread
            // 64 issues the copy
            auto issue = [&](int si) {
                const int c = si / np1, q = si - c * np1 + 1;
                if (c == 0) {
                    const long long t0 = spin_clock();
                    while (!(ready >> q & 1u)) {
                        const bool ok = lane >= 1 && lane < nparts && ld_acquire(flags + lane) == tag;
                        ready |= __ballot_sync(0xffffffffu, ok);
                        if (ready >> q & 1u) break;
                        int give_up = 0;
                        if (lane == 0) give_up = (*s_abort || spin_clock() - t0 > kWaitLimitCycles) ? 1 : 0;
                        if (__shfl_sync(0xffffffffu, give_up, 0)) {  // warp-uniform decision
                            if (lane == 0 && !*s_abort) {
                                *s_abort = 1;
                                atomicOr(status, kStatusTimeout);
                            }
                            return;
                        }
                        __nanosleep(32);
                    }
                }
                if (lane == 0) {
                    fence_proxy_async_global();
                    fence_proxy_async_smem();  // the slot was last touched by generic accesses
                    const int sl = si & (nsl - 1);
                    mbar_arrive_expect_tx(redbar + sl, slice_bytes);
                    bulk_load(red_stage + static_cast<size_t>(sl) * slice_bytes,
                              P.partials + static_cast<size_t>(c_first + q) * slot_floats +
                                  static_cast<size_t>(c) * 32 * kBM,
                              slice_bytes, redbar + sl);
                    inflight |= 1u << sl;
                }
            };
            // A 32-token tile (one chunk) skips the staging: each thread's 16 columns of its row of
            // every part come straight into registers, up to DP parts at a time once
            // their flags are seen, so the parts cost one round trip to L2 instead of a copy each
            // (the same sum, in the same order, bit for bit).
            constexpr bool direct = !WIDE;
            if (tr && threadIdx.x == 64) tr[kTrPartStored] = global_ns();
            // the QKV plan of a one-chunk tile does not need the sum: built while the parts arrive
            QkvPlan qpre;
            if constexpr (EPI == EPI_QKV) {
                if (direct) qpre = qkv_plan(ep, p, mt, nt * p.ntile, rt, esm, e, half);
            }
            if (ew == 0 && !direct) {
                if (nslices > 0) issue(0);
                if (nslices > 1 && nsl > 1) issue(1);
            }
            bool stop = false;
            int si = 0;
            for (int c = 0; c < nchunks && !stop; ++c) {
                if (direct) {
                    // The last part holds the tile's last k-blocks at the start of its CTA's range:
                    // it is fetched before the own accumulator is waited for (it usually finished
                    // earlier, and then costs nothing) and added after the middle parts, which
                    // follow in groups (the sum in part order).
                    if (!wait_parts(flags, nparts - 1, 1, tag, ew, lane, s_abort, status)) {
                        stop = true;
                        break;
                    }
                    const float4* srcl = reinterpret_cast<const float4*>(P.partials + static_cast<size_t>(c_last) * slot_floats);
                    float4 al[4];
#pragma unroll
                    for (int j = 0; j < 4; ++j) al[j] = __ldcg(srcl + static_cast<size_t>(half * 4 + j) * kBM + rt);
                    mbar_wait(&tfull[es.acc], es.acc_phase, s_abort, status);
                    if (named_bar_any(1, kEpiThreads, *s_abort != 0)) {
                        stop = true;
                        break;
                    }
                    if (tr && threadIdx.x == 64) {
                        tr[kTrAccReady] = global_ns();
                        tr[kTrTile] = static_cast<unsigned long long>(tile);
                    }
                    tc_fence_after();
                    tmem_ld_32x16(t_acc + static_cast<uint32_t>(half * 16), v);  // own (first) k-range
                    for (int q0 = 1; q0 < nparts - 1; q0 += DP) {
                        const int qn = min(DP, nparts - 1 - q0);
                        if (!wait_parts(flags, q0, qn, tag, ew, lane, s_abort, status)) {
                            stop = true;
                            break;
                        }
                        // L2 only (.cg): other CTAs wrote these lines, and the next launch writes
                        // the same slots again.  A group's loads go out unconditionally (the slot
                        // index held at the last part), its adds stop at the group's last part.
                        float4 a[DP][4];
#pragma unroll
                        for (int g = 0; g < DP; ++g) {
                            const float4* src = reinterpret_cast<const float4*>(
                                P.partials + static_cast<size_t>(min(c_first + q0 + g, c_last)) * slot_floats);
#pragma unroll
                            for (int j = 0; j < 4; ++j) a[g][j] = __ldcg(src + static_cast<size_t>(half * 4 + j) * kBM + rt);
                        }
#pragma unroll
                        for (int g = 0; g < DP; ++g)
                            if (g < qn) {
#pragma unroll
                                for (int j = 0; j < 4; ++j) {
                                    v[4 * j] += a[g][j].x;
                                    v[4 * j + 1] += a[g][j].y;
                                    v[4 * j + 2] += a[g][j].z;
                                    v[4 * j + 3] += a[g][j].w;
                                }
                            }
                    }
                    if (stop) break;
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        v[4 * j] += al[j].x;
                        v[4 * j + 1] += al[j].y;
                        v[4 * j + 2] += al[j].z;
                        v[4 * j + 3] += al[j].w;
                    }
                } else {
                    tmem_ld_32x16(t_acc + static_cast<uint32_t>(c * 32 + half * 16), v);  // own (first) k-range
                }
                // a wide residual tile's old rows of this chunk, loaded while its parts arrive
                float xw[kEpiGroup];
                if constexpr (EPI == EPI_RESID && WIDE) {
                    const int xrow = mt * kBM + rt;
#pragma unroll
                    for (int u = 0; u < kEpiGroup; ++u) {
                        const int xcol = nt * p.ntile + c * 32 + half * kEpiGroup + u;
                        xw[u] = (xrow < p.M && xcol < p.N) ? __ldcg(ep.out + static_cast<size_t>(xcol) * ep.ld_out + xrow)
                                                           : 0.0f;
                    }
                }
                for (int q = 1; !direct && q < nparts; ++q, ++si) {
                    const int sl = si & (nsl - 1);
                    mbar_wait(redbar + sl, (es.red_phase >> sl) & 1u, s_abort, status);
                    es.red_phase ^= 1u << sl;
                    if (threadIdx.x == 64) inflight &= ~(1u << sl);
                    const float4* src = reinterpret_cast<const float4*>(red_stage + static_cast<size_t>(sl) * slice_bytes);
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const float4 a = src[(half * 4 + j) * kBM + rt];
                        v[4 * j] += a.x;
                        v[4 * j + 1] += a.y;
                        v[4 * j + 2] += a.z;
                        v[4 * j + 3] += a.w;
                    }
                    if (named_bar_any(1, kEpiThreads, *s_abort != 0)) {  // the slot is free again (or the launch failed)
                        stop = true;
                        break;
                    }
                    if (ew == 0 && si + nsl < nslices) issue(si + nsl);
                }
                if (stop) break;
                if (tr && threadIdx.x == 64 && c == 0) {
                    tr[kTrTicket] = global_ns();
                    tr[kTrReduced] = global_ns();
                    tr[kTrIsLast] = 1;
                }
                // the compact epilogue on the sum in registers (the residual's first pass leaves the
                // new residual in the still owned accumulator, for the second)
                epilogue_c32<EPI, kPass1>(ep, p, mt, nt * p.ntile + c * 32, c * 32, rt,
                                          t_acc + static_cast<uint32_t>(c * 32),
                                          t_x ? t_x + static_cast<uint32_t>(c * 32) : 0u, esm, e, half, quarter, lane,
                                          status, v, (EPI == EPI_QKV && direct) ? &qpre : nullptr,
                                          EPI == EPI_RESID && WIDE ? xw : nullptr);
            }
            if (threadIdx.x == 64) {
                if (stop) {  // let copies in flight land before the shared memory is released
                    const long long t0 = spin_clock();
                    for (int sl = 0; sl < nsl; ++sl)
                        while ((inflight >> sl & 1u) && !mbar_try_wait(redbar + sl, (es.red_phase >> sl) & 1u) &&
                               spin_clock() - t0 < kWaitLimitCycles) {
                        }
                } else {
                    for (int q = 1; q < nparts; ++q) flags[q] = 0;  // ready for the next launch
                }
            }
            if (stop) {
                cp_async_wait<0>();
                return;
            }
        }
        if (tr && threadIdx.x == 64) tr[kTrEpiPass1] = global_ns();
        if (finisher && P.done) {  // publish the finished tile to the next phase's operand producer
            named_bar(1, kEpiThreads);
            if (threadIdx.x == 64) {
                st_release(&P.done[mt * p.n_tiles + nt], tag);
                if (tr) tr[kTrPublished] = global_ns();
            }
        }
        if constexpr (EPI == EPI_RESID) {
            if (finisher) {  // then the fp32 residual and the RMSNorm sums, for the later phases' epilogues
                for (int c = 0; c < nchunks; ++c)
                    epilogue_c32<EPI, 2>(ep, p, mt, nt * p.ntile + c * 32, c * 32, rt,
                                         t_acc + static_cast<uint32_t>(c * 32), 0u, esm, e, half, quarter,
                                         lane, status);
                if (P.done2) {
                    named_bar(1, kEpiThreads);
                    if (threadIdx.x == 64) st_release(&P.done2[mt * p.n_tiles + nt], tag);
                }
            }
        }
        if (finisher) {
            tc_fence_before();
            mbar_arrive(&tempty[es.acc]);
        }
        if (++es.acc == 2) {
            es.acc = 0;
            es.acc_phase ^= 1u;
        }
        it = tile * p.kb + k_hi;
    }
    cp_async_wait<0>();
    if (tr && threadIdx.x == 64) tr[kTrEpiDone] = global_ns();
}

template <int DP, bool WIDE>
__device__ __forceinline__ void chain_epilogue_dispatch(const ChainArgs& ca, int ph, int tag, uint8_t* red_stage,
                                                        uint64_t* tfull, uint64_t* tempty, uint64_t* redbar,
                                                        volatile int* s_abort, uint32_t tmem_base, const EpiSmem& esm,
                                                        ChainEpiState& es) {
    switch (ca.ph[ph].epi) {
        case EPI_F32:
            chain_phase_epilogue<EPI_F32, DP, WIDE>(ca, ph, tag, red_stage, tfull, tempty, redbar, s_abort, tmem_base, esm, es);
            break;
        case EPI_RESID:
            chain_phase_epilogue<EPI_RESID, DP, WIDE>(ca, ph, tag, red_stage, tfull, tempty, redbar, s_abort, tmem_base, esm, es);
            break;
        case EPI_QKV:
            chain_phase_epilogue<EPI_QKV, DP, WIDE>(ca, ph, tag, red_stage, tfull, tempty, redbar, s_abort, tmem_base, esm, es);
            break;
        case EPI_SWIGLU:
            chain_phase_epilogue<EPI_SWIGLU, DP, WIDE>(ca, ph, tag, red_stage, tfull, tempty, redbar, s_abort, tmem_base, esm, es);
            break;
        default:
            chain_phase_epilogue<EPI_LMHEAD, DP, WIDE>(ca, ph, tag, red_stage, tfull, tempty, redbar, s_abort, tmem_base, esm, es);
            break;
    }
}

// Expand row t of one 4-bit weight tile (see kQ4TileBytes) into its 64 bf16 weights, as 32
// pairs o[c][j] = (k = 8c + 2j, 8c + 2j + 1), each weight bf16(d * (q - 8)).  128 + q is built as
// a bf16 bit pattern (exponent of 128, q in the low mantissa bits), 136 is subtracted exactly
// and the scale applied with one correctly rounded bf16 multiply.
__device__ __forceinline__ void q4_expand(const uint8_t* __restrict__ raw, int t, uint32_t (&o)[8][4]) {
    const uint32_t* codes = reinterpret_cast<const uint32_t*>(raw);
    const uint16_t* sc = reinterpret_cast<const uint16_t*>(raw + 4096);
    // every load first (the raw slot and the A stage may both be shared memory: loads issued
    // after a store could not be moved above it), then the arithmetic of all eight chunks
    uint32_t w[8];
#pragma unroll
    for (int c = 0; c < 8; ++c) w[c] = codes[c * 128 + t];
    const uint32_t s0 = sc[t], s1 = sc[128 + t];
    const uint32_t d0 = s0 | (s0 << 16), d1 = s1 | (s1 << 16);  // (d, d) as bf16x2, per block of 32
#pragma unroll
    for (int c = 0; c < 8; ++c) {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            uint32_t v, x;
            // (w >> 4j) & 0x000F000F | 0x43004300: the bf16 pair (128 + q, 128 + q') of two columns
            asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(v) : "r"(w[c] >> (4 * j)), "r"(0x000F000Fu), "r"(0x43004300u));
            asm("sub.rn.bf16x2 %0, %1, %2;" : "=r"(x) : "r"(v), "r"(0x43084308u));           // - (136, 136): exact
            asm("mul.rn.bf16x2 %0, %1, %2;" : "=r"(o[c][j]) : "r"(x), "r"(c < 4 ? d0 : d1));  // * d: one rounding
        }
    }
}

// ... into the 128-byte-swizzled K-major bf16 image in shared memory the UMMA descriptor reads
// (thread t of the 128 writes row t)
__device__ __forceinline__ void q4_expand_row(const uint8_t* __restrict__ raw, uint8_t* __restrict__ dst_tile, int t) {
    uint32_t o[8][4];
    q4_expand(raw, t, o);
    uint8_t* row = dst_tile + t * 128;
#pragma unroll
    for (int c = 0; c < 8; ++c)
        *reinterpret_cast<uint4*>(row + ((c ^ (t & 7)) << 4)) = make_uint4(o[c][0], o[c][1], o[c][2], o[c][3]);
}

// ... or into tensor memory, row r at lane r: 64 weights in 32 columns from taddr, the pair of
// k = 2i, 2i + 1 in column i (the layout of an MMA's A operand read from tensor memory); the
// calling warp's lanes are rows 32 (warp % 4) .. +31.  The caller waits for the store
// (tcgen05.wait::st) before it publishes the stage.
__device__ __forceinline__ void tmem_st_row64(uint32_t taddr, const uint32_t (&o)[8][4]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
        "%14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
        "r"(o[0][0]), "r"(o[0][1]), "r"(o[0][2]), "r"(o[0][3]), "r"(o[1][0]), "r"(o[1][1]), "r"(o[1][2]), "r"(o[1][3]),
        "r"(o[2][0]), "r"(o[2][1]), "r"(o[2][2]), "r"(o[2][3]), "r"(o[3][0]), "r"(o[3][1]), "r"(o[3][2]), "r"(o[3][3]),
        "r"(o[4][0]), "r"(o[4][1]), "r"(o[4][2]), "r"(o[4][3]), "r"(o[5][0]), "r"(o[5][1]), "r"(o[5][2]), "r"(o[5][3]),
        "r"(o[6][0]), "r"(o[6][1]), "r"(o[6][2]), "r"(o[6][3]), "r"(o[7][0]), "r"(o[7][1]), "r"(o[7][2]), "r"(o[7][3])
        : "memory");
}

// n (1 or 2) consecutive tiles of one raw slot into consecutive 32-column groups from taddr
__device__ __forceinline__ void q4_expand_tmem(const uint8_t* __restrict__ raw, int r, uint32_t taddr, int n) {
    uint32_t o[8][4];
    q4_expand(raw, r, o);
    tmem_st_row64(taddr, o);
    if (n == 2) {
        q4_expand(raw + kQ4TileBytes, r, o);
        tmem_st_row64(taddr + 32, o);
    }
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

template <bool Q4>
__global__ void __launch_bounds__(Q4 ? kChainThreadsQ4 : kChainThreads, 1)
    k_chain(const __grid_constant__ ChainMaps maps, const __grid_constant__ ChainArgs ca) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int S = ca.stages;
    const int R = Q4 ? ca.raw_stages : 0;
    // 4-bit weights: the operand (B) tiles have a ring of their own, deeper than the A stages
    const int SB = Q4 ? ca.b_stages : S;
    const uint32_t b_bytes = static_cast<uint32_t>(ca.ntile) * kBK * 2;
    // 4-bit weights with the A stages in tensor memory (ca.a_tmem): no shared A stages, and a
    // pipeline stage holds up to two consecutive k-blocks of one tile (kper): one wait, one
    // arrival and one commit per role for both.  A tile's run of k-blocks in this CTA's range
    // is cut into pairs from its start; an odd run ends with a stage of one.
    const bool a_tm = Q4 && ca.a_tmem;
    const int kper = a_tm ? 2 : 1;
    const uint32_t b_slot = b_bytes * static_cast<uint32_t>(kper);
    const uint32_t raw_slot = kQ4TileBytes * static_cast<uint32_t>(kper);
    uint8_t* sA = smem;
    uint8_t* sB = sA + (a_tm ? 0 : static_cast<size_t>(S) * kABytes);
    uint8_t* sRaw = sB + static_cast<size_t>(SB) * b_slot;  // 4-bit weight tiles (Q4)
    uint8_t* red_stage = sRaw + static_cast<size_t>(R) * raw_slot;
    float* tail = reinterpret_cast<float*>(red_stage + ca.red_bytes + ca.stg_bytes);
    EpiSmem esm;
    esm.rs = tail;
    esm.red = tail + 256;
    esm.kvs = reinterpret_cast<int*>(tail + 256 + 1024);
    esm.theta = tail + 256 + 1024 + 256;
    esm.stg = ca.stg_bytes ? red_stage + ca.red_bytes : red_stage;
    float* after = tail + 256 + 1024 + 256 + 128;
    uint64_t* full = reinterpret_cast<uint64_t*>(after);
    uint64_t* empty = full + S;
    uint64_t* tfull = empty + S;
    uint64_t* tempty = tfull + 2;
    uint64_t* drain = tempty + 2;
    uint64_t* redbar = drain + 1;  // the partial staging slots (one or two)
    uint64_t* rfull = redbar + 2;  // raw 4-bit tiles (Q4): arrived / read
    uint64_t* rempty = rfull + R;
    uint64_t* bfull = rempty + R;  // operand tiles of the 4-bit kernel: arrived / consumed
    uint64_t* bempty = bfull + (Q4 ? SB : 0);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bempty + (Q4 ? SB : 0));
    volatile int* s_abort = reinterpret_cast<volatile int*>(tmem_slot + 1);
    int* s_rows = reinterpret_cast<int*>(tmem_slot + 2);
    esm.rows = s_rows;
    int* status = ca.status;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        pdl_launch_dependents();
        for (int s = 0; s < S; ++s) {
            // Q4: one arrival per dequantizing warp (the operand has barriers of its own)
            mbar_init(&full[s], Q4 ? kDeqWarps : 1);
            mbar_init(&empty[s], 1);
        }
        for (int r = 0; r < R; ++r) {
            mbar_init(&rfull[r], 1);
            mbar_init(&rempty[r], kDeqWarps);
        }
        if (Q4)
            for (int b = 0; b < SB; ++b) {
                mbar_init(&bfull[b], 1);
                mbar_init(&bempty[b], 1);
            }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&tfull[a], 1);
            mbar_init(&tempty[a], kEpiThreads);
        }
        mbar_init(drain, 1);
        mbar_init(&redbar[0], 1);
        mbar_init(&redbar[1], 1);
        *s_abort = 0;
        int rows = -1;
        if (ca.dyn_rows) {
            pdl_wait();  // the count is written by the preceding launch
            rows = max(*ca.dyn_rows, 0);
        }
        *s_rows = rows;
        mbar_fence_init();
    }
    if (warp == 0 && lane == 0) {
        for (int ph = 0; ph < ca.n_phases; ++ph)
            if (!ca.ph[ph].w_tiles) tma_prefetch_desc(&maps.w[ph]);
    }
    if (warp == 6 && lane == 0) {
        for (int ph = 0; ph < ca.n_phases; ++ph) tma_prefetch_desc(&maps.x[ph]);
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, ca.tmem_cols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    const int acc_cols = ca.acc_cols;
    const int rows = *s_rows;

    if (warp == 0) {
        // ---------------------------------------------------------- weight producer
        if (lane == 0) {
            const uint64_t pol_w = policy_evict_first();
            int stage = 0;
            uint32_t par = 0;
            uint32_t pending = 0, pend_par = 0;
            constexpr uint32_t tile_bytes = Q4 ? kQ4TileBytes : kABytes;
            for (int ph = 0; ph < ca.n_phases && !*s_abort; ++ph) {
                const GemmPlan p = phase_plan(ca.ph[ph], rows);
                if (static_cast<int>(blockIdx.x) >= p.grid) continue;
                const int it0 = static_cast<int>(range_begin(blockIdx.x, p.total, p.grid));
                const int it1 = static_cast<int>(range_begin(blockIdx.x + 1, p.total, p.grid));
                unsigned long long* tr = ca.ph[ph].ep.trace ? ca.ph[ph].ep.trace + static_cast<size_t>(blockIdx.x) * kTrSlots : nullptr;
                if (tr) tr[kTrStart] = global_ns();
                // (m-tile, k-block) walked incrementally: no division in the loop
                int tile = it0 / p.kb, k = it0 - tile * p.kb;
                int nt = tile / p.m_tiles, mt = tile - nt * p.m_tiles;
                const char* wt = reinterpret_cast<const char*>(ca.ph[ph].w_tiles);
                size_t woff = (static_cast<size_t>(mt) * p.kb + k) * tile_bytes;  // tile-major: (mt*kb + k) tiles
                for (int it = it0; it < it1;) {
                    const int n = (a_tm && k + 1 < p.kb && it + 1 < it1) ? 2 : 1;  // k-blocks of this stage
                    if constexpr (Q4) {
                        // the raw tile goes to its own ring; the dequantizing warps fill the A stage.
                        // A stages in tensor memory: raw slot s belongs to A stage s, and is free
                        // again once the MMAs that read that stage are done; a pair of tiles of
                        // one row block is one contiguous copy
                        if (!mbar_wait(a_tm ? &empty[stage] : &rempty[stage], par ^ 1u, s_abort, status)) break;
                        mbar_arrive_expect_tx(&rfull[stage], n * kQ4TileBytes);
                        bulk_load_hint(sRaw + static_cast<size_t>(stage) * raw_slot, wt + woff, n * kQ4TileBytes,
                                       &rfull[stage], pol_w);
                    } else {
                        if (!mbar_wait(&empty[stage], par ^ 1u, s_abort, status)) break;
                        mbar_arrive_expect_tx(&full[stage], kABytes + b_bytes);
                        if (wt)
                            bulk_load_hint(sA + static_cast<size_t>(stage) * kABytes, wt + woff, kABytes,
                                           &full[stage], pol_w);
                        else
                            tma_load_2d(sA + static_cast<size_t>(stage) * kABytes, &maps.w[ph], k * kBK, mt * kBM,
                                        &full[stage], pol_w);
                    }
                    pending |= 1u << stage;
                    pend_par = (pend_par & ~(1u << stage)) | (par << stage);
                    if (++stage == (Q4 ? R : S)) {
                        stage = 0;
                        par ^= 1u;
                    }
                    it += n;
                    woff += static_cast<size_t>(n) * tile_bytes;
                    k += n;
                    if (k == p.kb) {
                        k = 0;
                        if (++mt == p.m_tiles) {
                            mt = 0;
                            woff = 0;
                            ++nt;
                        }
                    }
                }
            }
            if (*s_abort) {
                // let the copies in flight land before the CTA's shared memory is released (a
                // stage whose operand was never issued does not complete: one deadline for all)
                const long long t0 = spin_clock();
                for (int s = 0; s < (Q4 ? R : S); ++s) {
                    if (!(pending >> s & 1u)) continue;
                    uint64_t* bar = Q4 ? &rfull[s] : &full[s];
                    while (!mbar_try_wait(bar, (pend_par >> s) & 1u) && spin_clock() - t0 < kWaitLimitCycles) {
                    }
                }
            }
        }
    } else if (warp == 6) {
        // ---------------------------------------------------------- operand producer
        // The whole warp runs the loop: its slot waits are voted warp-wide, so that the copy
        // coordinates stay warp-uniform values, one elected lane issues the copies, and the
        // completion flags of the producing tiles are polled 32 at a time (one round trip
        // covers the next 32).
        const uint64_t pol_x = policy_evict_last();
        pdl_wait();
        const int tag = chain_tag(ca);
        const bool leader = elect_one();
        const int urows = __shfl_sync(0xffffffffu, rows, 0);
        int stage = 0;
        uint32_t par = 0;
        uint32_t bpend = 0, bpend_par = 0;  // Q4: operand copies issued (for the drain on abort)
        bool stop = false;
        if (ca.gate) {  // the bounded-wait test hook (see ChainArgs::gate)
            int open = 1;
            if (lane == 0) open = wait_flag(ca.gate, tag, s_abort, status) ? 1 : 0;
            stop = __shfl_sync(0xffffffffu, open, 0) == 0;  // warp-uniform decision
        }
        for (int ph = 0; ph < ca.n_phases && !stop; ++ph) {
            const ChainPhase& P = ca.ph[ph];
            const GemmPlan p = phase_plan(P, urows);
            if (static_cast<int>(blockIdx.x) >= p.grid) continue;
            const int it0 = static_cast<int>(range_begin(blockIdx.x, p.total, p.grid));
            const int it1 = static_cast<int>(range_begin(blockIdx.x + 1, p.total, p.grid));
            const int* dep = (ph > 0 && P.dep_rows > 0) ? ca.ph[ph - 1].done : nullptr;
            const int dep_tiles = dep ? ca.ph[ph - 1].p.m_tiles : 0;
            const int dep_shift = dep ? 31 - __clz(P.dep_rows) : 0;  // dep_rows is a power of two
            // completion of the previous phase's tiles for token tile mine_nt, as far as seen:
            // lane l, bit w = tile 32w + l (a flag, once complete, stays so for the launch)
            uint32_t mine = 0;
            int mine_nt = -1;
            int tile = it0 / p.kb, k = it0 - tile * p.kb;
            int nt = tile / p.m_tiles, mt = tile - nt * p.m_tiles;
            for (int it = it0; it < it1;) {
                const int n = (a_tm && k + 1 < p.kb && it + 1 < it1) ? 2 : 1;  // k-blocks of this stage
                if (!__all_sync(0xffffffffu, mbar_wait(Q4 ? &bempty[stage] : &empty[stage], par ^ 1u, s_abort, status))) {
                    stop = true;
                    break;
                }
                for (int j = 0; dep && j < n; ++j) {
                    const int pmt = ((k + j) * kBK) >> dep_shift;
                    if (nt != mine_nt) {
                        mine = 0;
                        mine_nt = nt;
                    }
                    if (!(__shfl_sync(0xffffffffu, mine, pmt & 31) >> (pmt >> 5) & 1u)) {
                        // poll the 32 producing tiles around pmt (one acquire load per lane) until
                        // pmt is complete; what is seen complete is kept for the later k-blocks
                        const int w = pmt >> 5;
                        const long long t0 = spin_clock();
                        for (;;) {
                            const int i = w * 32 + lane;
                            const bool ok = i >= dep_tiles || ld_acquire(dep + i * p.n_tiles + nt) == tag;
                            const uint32_t seen = __ballot_sync(0xffffffffu, ok);
                            mine |= ((seen >> lane) & 1u) << w;
                            if (seen >> (pmt & 31) & 1u) {
                                fence_proxy_async_global();  // generic-proxy writes of other CTAs -> these TMA reads
                                break;
                            }
                            int give_up = 0;
                            if (lane == 0) give_up = (*s_abort || spin_clock() - t0 > kWaitLimitCycles) ? 1 : 0;
                            if (__shfl_sync(0xffffffffu, give_up, 0)) {  // warp-uniform decision
                                if (lane == 0 && !*s_abort) {
                                    *s_abort = 1;
                                    atomicOr(status, kStatusTimeout);
                                }
                                stop = true;
                                break;
                            }
                            __nanosleep(32);
                        }
                        if (stop) break;
                    }
                }
                if (stop) break;
                if (leader) {
                    uint64_t* fb = Q4 ? &bfull[stage] : &full[stage];
                    if constexpr (Q4) {  // its own barrier; the A part of the stage arrives by the dequantizers
                        mbar_arrive_expect_tx(fb, n * b_bytes);
                        bpend |= 1u << stage;
                        bpend_par = (bpend_par & ~(1u << stage)) | (par << stage);
                    }
                    for (int j = 0; j < n; ++j)
                        tma_load_2d(sB + static_cast<size_t>(stage) * b_slot + static_cast<size_t>(j) * b_bytes, &maps.x[ph],
                                    (k + j) * kBK, nt * ca.ntile, fb, pol_x);
                }
                __syncwarp();
                if (++stage == SB) {
                    stage = 0;
                    par ^= 1u;
                }
                it += n;
                k += n;
                if (k == p.kb) {
                    k = 0;
                    if (++mt == p.m_tiles) {
                        mt = 0;
                        ++nt;
                    }
                }
            }
        }
        if constexpr (Q4) {
            // the operand ring is this warp's alone: on an abort, let its copies in flight land
            // before the CTA's shared memory is released (one deadline for all)
            if (leader && *s_abort) {
                const long long t0 = spin_clock();
                for (int b = 0; b < SB; ++b)
                    while ((bpend >> b & 1u) && !mbar_try_wait(&bfull[b], (bpend_par >> b) & 1u) &&
                           spin_clock() - t0 < kWaitLimitCycles) {
                    }
            }
        }
    } else if (Q4 && warp >= kDeqWarp0) {
        // ---------------------------------------------------------- dequantizers (4-bit weights)
        // Every stage: wait for its raw tiles (shared A stages: and for the stage to be free),
        // expand them, make the writes visible to the tensor cores, and arrive (one arrival per
        // warp) on the stage's full barrier (shared A stages: and on the raw slot's empty
        // barrier).  Shared A stages: thread t writes row t; A stages in tensor memory: a warp
        // writes the rows of its TMEM lane quarter, 32 (warp % 4) + lane.
        const int t = a_tm ? (warp & 3) * 32 + lane : threadIdx.x - kDeqWarp0 * 32;
        const uint32_t a_lane = static_cast<uint32_t>((warp & 3) * 32) << 16;
        int stage = 0, rs = 0;
        uint32_t par = 0, rpar = 0;
        bool stop = false;
        for (int ph = 0; ph < ca.n_phases && !stop; ++ph) {
            const GemmPlan p = phase_plan(ca.ph[ph], rows);
            if (static_cast<int>(blockIdx.x) >= p.grid) continue;
            const int it0 = static_cast<int>(range_begin(blockIdx.x, p.total, p.grid));
            const int it1 = static_cast<int>(range_begin(blockIdx.x + 1, p.total, p.grid));
            if (a_tm) {
                // raw slot and A stage share one index: the raw tiles' arrival implies that the
                // MMAs which read the stage's previous tiles are done (the producer loaded them
                // only after their commit), so one wait and one arrival per stage
                int k = it0 - (it0 / p.kb) * p.kb;
                for (int it = it0; it < it1;) {
                    const int n = (k + 1 < p.kb && it + 1 < it1) ? 2 : 1;  // k-blocks of this stage
                    if (!mbar_wait(&rfull[stage], par, s_abort, status)) {
                        stop = true;
                        break;
                    }
                    tc_fence_after();
                    q4_expand_tmem(sRaw + static_cast<size_t>(stage) * raw_slot, t,
                                   tmem_base + a_lane + static_cast<uint32_t>(ca.a_col0 + stage * kBK), n);
                    tc_fence_before();  // the tensor-memory writes -> the MMA issuer's wait
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&full[stage]);
                    if (++stage == S) {
                        stage = 0;
                        par ^= 1u;
                    }
                    it += n;
                    k += n;
                    if (k == p.kb) k = 0;
                }
                continue;
            }
            for (int it = it0; it < it1; ++it) {
                if (!mbar_wait(&rfull[rs], rpar, s_abort, status) || !mbar_wait(&empty[stage], par ^ 1u, s_abort, status)) {
                    stop = true;
                    break;
                }
                q4_expand_row(sRaw + static_cast<size_t>(rs) * kQ4TileBytes, sA + static_cast<size_t>(stage) * kABytes, t);
                fence_proxy_async_smem();  // generic writes (and the raw reads) -> async-proxy accesses
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive(&full[stage]);
                    mbar_arrive(&rempty[rs]);
                }
                if (++stage == S) {
                    stage = 0;
                    par ^= 1u;
                }
                if (++rs == R) {
                    rs = 0;
                    rpar ^= 1u;
                }
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------------- MMA issuer
        // The whole warp runs the loop (its waits and their outcomes voted warp-wide), so that
        // the tensor-memory addresses and shared-memory descriptors are warp-uniform values;
        // one elected lane issues the MMAs and the commits.
        const bool leader = elect_one();
        const uint32_t tbase = __shfl_sync(0xffffffffu, tmem_base, 0);
        const int urows = __shfl_sync(0xffffffffu, rows, 0);
        const uint32_t idesc = umma_idesc_bf16(kBM, ca.ntile);
        int stage = 0, bstage = 0;  // A stage; Q4: the operand's own ring
        uint32_t par = 0, bpar = 0;
        int acc = 0;
        uint32_t acc_phase = 0;
        bool issued = false, stop = false;
        for (int ph = 0; ph < ca.n_phases && !stop; ++ph) {
            const GemmPlan p = phase_plan(ca.ph[ph], urows);
            if (static_cast<int>(blockIdx.x) >= p.grid) continue;
            const long long it0 = range_begin(blockIdx.x, p.total, p.grid);
            const long long it1 = range_begin(blockIdx.x + 1, p.total, p.grid);
            unsigned long long* tr =
                (leader && ca.ph[ph].ep.trace) ? ca.ph[ph].ep.trace + static_cast<size_t>(blockIdx.x) * kTrSlots : nullptr;
            bool first = true;
            for (long long it = it0; it < it1;) {
                const long long tile = it / p.kb;
                const int k_lo = static_cast<int>(it - tile * p.kb);
                const long long tend = (tile + 1) * p.kb;
                const int k_hi = static_cast<int>((it1 < tend ? it1 : tend) - tile * p.kb);
                if (__any_sync(0xffffffffu, *s_abort != 0) ||
                    !__all_sync(0xffffffffu, mbar_wait(&tempty[acc], acc_phase ^ 1u, s_abort, status))) {
                    stop = true;
                    break;
                }
                tc_fence_after();
                const uint32_t d_tmem = tbase + static_cast<uint32_t>(acc * acc_cols);
                for (int k = k_lo; k < k_hi;) {
                    const int n = (a_tm && k + 1 < k_hi) ? 2 : 1;  // k-blocks of this stage
                    const bool got = mbar_wait(&full[stage], par, s_abort, status) &&
                                     (!Q4 || mbar_wait(&bfull[bstage], bpar, s_abort, status));
                    if (!__all_sync(0xffffffffu, got)) {
                        stop = true;
                        break;
                    }
                    if (tr && first) tr[kTrFirstData] = global_ns();
                    first = false;
                    tc_fence_after();
                    const uint8_t* b_st = sB + static_cast<size_t>(Q4 ? bstage : stage) * b_slot;
                    const uint64_t bdesc = sw128_kmajor_desc(smem_u32(b_st));
                    if (leader) {
                        if (a_tm) {  // A: 8 tensor-memory columns per 16-wide K step, 32 per k-block
                            const uint32_t a_t = tbase + static_cast<uint32_t>(ca.a_col0 + stage * kBK);
#pragma unroll
                            for (int kk = 0; kk < kBK / 16; ++kk)
                                umma_bf16_tmem_a(d_tmem, a_t + static_cast<uint32_t>(kk * 8), bdesc + 2ull * kk, idesc,
                                                 (k > k_lo || kk > 0) ? 1u : 0u);
                            if (n == 2) {
                                const uint64_t bdesc1 = sw128_kmajor_desc(smem_u32(b_st + b_bytes));
#pragma unroll
                                for (int kk = 0; kk < kBK / 16; ++kk)
                                    umma_bf16_tmem_a(d_tmem, a_t + static_cast<uint32_t>(32 + kk * 8), bdesc1 + 2ull * kk,
                                                     idesc, 1u);
                            }
                        } else {
                            const uint64_t adesc = sw128_kmajor_desc(smem_u32(sA + static_cast<size_t>(stage) * kABytes));
#pragma unroll
                            for (int kk = 0; kk < kBK / 16; ++kk)
                                umma_bf16(d_tmem, adesc + 2ull * kk, bdesc + 2ull * kk, idesc,
                                          (k > k_lo || kk > 0) ? 1u : 0u);
                        }
                        umma_commit(&empty[stage]);
                        if constexpr (Q4) umma_commit(&bempty[bstage]);
                    }
                    __syncwarp();
                    issued = true;
                    if (++stage == S) {
                        stage = 0;
                        par ^= 1u;
                    }
                    if constexpr (Q4) {
                        if (++bstage == SB) {
                            bstage = 0;
                            bpar ^= 1u;
                        }
                    }
                    k += n;
                }
                if (stop) break;
                if (leader) umma_commit(&tfull[acc]);
                __syncwarp();
                if (++acc == 2) {
                    acc = 0;
                    acc_phase ^= 1u;
                }
                it = tile * p.kb + k_hi;
            }
            if (tr) tr[kTrLastData] = global_ns();
        }
        if (__any_sync(0xffffffffu, *s_abort != 0) && issued) {
            if (leader) {  // the MMAs in flight finish before tensor memory is released
                umma_commit(drain);
                const long long t0 = spin_clock();
                while (!mbar_try_wait(drain, 0) && spin_clock() - t0 < kWaitLimitCycles) {
                }
            }
            __syncwarp();
        }
    } else {
        // ---------------------------------------------------------- epilogue
        pdl_wait();
        const int tag = chain_tag(ca);
        ChainEpiState es{0, 0u, 0u};
        // split 32-token tiles: parts whose rows are loaded into registers at once (the 4-bit
        // kernel's smaller register budget takes two)
        constexpr int kDP = Q4 ? 2 : 4;
        for (int ph = 0; ph < ca.n_phases; ++ph) {  // on abort every phase returns at its first barrier
            if (ca.ntile == 32)
                chain_epilogue_dispatch<kDP, false>(ca, ph, tag, red_stage, tfull, tempty, redbar, s_abort, tmem_base,
                                                    esm, es);
            else
                chain_epilogue_dispatch<kDP, true>(ca, ph, tag, red_stage, tfull, tempty, redbar, s_abort, tmem_base,
                                                   esm, es);
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) {
        __syncwarp();
        tmem_dealloc(tmem_base, ca.tmem_cols);
    }
}

// ------------------------------------------------------------------ host side
static int pow2ceil(int x) {
    int p = 32;
    while (p < x) p <<= 1;
    return p;
}

GemmPlan gemm_plan(int M, int N, int K, int grid_max, int epi) {
    GemmPlan p{};
    p.M = M;
    p.N = N;
    p.K = K;
    p.n_tiles = (N + 255) / 256;
    const int per = (N + p.n_tiles - 1) / p.n_tiles;
    p.ntile = ((per + 31) / 32) * 32;
    p.m_tiles = (M + kBM - 1) / kBM;
    p.kb = (K + kBK - 1) / kBK;
    p.total = static_cast<long long>(p.m_tiles) * p.n_tiles * p.kb;
    p.grid = static_cast<int>(p.total < grid_max ? p.total : grid_max);
    // at least ceil(kb/30) iterations per CTA, so a tile has at most 31 parts (one completion
    // flag each in its 32-int line)
    const long long min_iters = (p.kb + 29) / 30;
    if (p.grid > p.total / min_iters) p.grid = static_cast<int>(p.total / min_iters);
    if (p.grid < 1) p.grid = 1;
    p.pdl = true;
    return p;
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn get_encode() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(ptr);
    }
    return fn;
}

bool make_tmap_bf16(CUtensorMap* tm, const void* ptr, uint64_t rows, uint64_t cols, uint32_t box_rows) {
    EncodeTiledFn enc = get_encode();
    if (!enc) return false;
    if ((reinterpret_cast<uintptr_t>(ptr) & 15) || ((cols * 2) & 15) || box_rows == 0 || box_rows > 256) return false;
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {cols * 2};
    cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

cudaError_t gemm_init_attrs() { return chain_init_attrs(); }

// One projection = a chain of one phase.
cudaError_t gemm_launch(int epi, const GemmPlan& p, const CUtensorMap& tmW, const CUtensorMap& tmX,
                        const EpiArgs& ep, const Scratch& scr, int* status, cudaStream_t st, const int* gate) {
    if (gemm_partial_floats(p) > scr.partial_floats ||
        static_cast<long long>(p.m_tiles) * p.n_tiles * kTicketStride > scr.counter_len)
        return cudaErrorInvalidValue;
    ChainArgs ca{};
    ca.n_phases = 1;
    ca.status = status;
    ca.tag_add = 1;
    ca.gate = gate;
    ChainPhase& P = ca.ph[0];
    P.p = p;
    P.ep = ep;
    P.epi = epi;
    P.partials = scr.partials;
    P.tickets = scr.counters;
    if (!chain_plan(ca, g_stream_budget)) return cudaErrorInvalidValue;
    ChainMaps m;
    m.w[0] = tmW;
    m.x[0] = tmX;
    return chain_launch(m, ca, st, p.pdl);
}

void set_stream_smem(bool coresident) { g_stream_budget = coresident ? kChainSmemShared : kChainSmemFull; }

static bool g_pdl = true;
void set_pdl(bool on) { g_pdl = on; }
bool pdl_enabled() { return g_pdl; }


bool chain_plan(ChainArgs& ca, int smem_budget) {
    if (ca.n_phases < 1 || ca.n_phases > kMaxPhases) return false;
    const int ntile = ca.ph[0].p.ntile;
    int grid = 0;
    for (int i = 0; i < ca.n_phases; ++i) {
        const GemmPlan& p = ca.ph[i].p;
        if (p.ntile != ntile || p.N != ca.ph[0].p.N) return false;
        grid = grid > p.grid ? grid : p.grid;
    }
    for (int i = 1; i < ca.n_phases; ++i)
        if (ca.ph[i].dep_rows > 0 && ca.ph[i - 1].p.m_tiles > kMaxDepTiles) return false;
    const bool c32 = ntile == 32;
    // wider token tiles are tensor-bound: the deepest ring (the attention CTAs' room matters
    // only to the batch-1 weight stream)
    if (!c32) smem_budget = kFullSmem;
    ca.grid = grid;
    ca.ntile = ntile;
    ca.acc_cols = c32 ? 32 : pow2ceil(ntile);
    ca.x_cols = ntile <= 128 ? ntile : 0;  // staged residual (none for 256-token tiles: TMEM is full)
    ca.tmem_cols = pow2ceil(2 * ca.acc_cols + ca.x_cols);
    // Partial slices staged for the finisher of a split tile of several 32-token chunks: two in
    // flight, one for 256-token tiles (their ring needs the room: the tensor cores keep busy
    // with 4 stages of 256 tokens, not with 3); for 32-token chains, whose finishers load the
    // parts straight into registers, one slot that is the output staging.
    ca.red_bytes = (c32 || ntile > 128 ? 1 : 2) * 32 * kBM * 4;
    const int stage_bytes = static_cast<int>(kABytes) + ntile * kBK * 2;
    // tiles of more than one 32-token chunk: their own 8 KB for the bf16 output staging
    ca.stg_bytes = c32 ? 0 : 32 * kBM * 2;
    const int fixed0 = 1024 + (256 + 1024 + 256 + 128) * 4 + ca.red_bytes + ca.stg_bytes + 7 * 8 + 16;
    if (ca.q4) {
        // 4-bit weights (480 threads: no room beside the CTA for another one, so all of shared
        // memory): raw 4.5 KB tiles, a few bf16 A stages the dequantizers fill (in tensor memory
        // where it has the room, else shared), and a ring of operand tiles of its own, as deep as
        // what is left allows (2 .. 24)
        const int kRaw[3] = {12, 8, 6}, kA[3] = {4, 3, 2};
        const int b_stage = ntile * kBK * 2 + 16;
        const int a_col0 = 2 * ca.acc_cols + ca.x_cols;
        // A stages in tensor memory where it holds at least 4 stages of two k-blocks (64 columns
        // each): then raw slots (two tiles each) and A stages are one ring of up to 6 stages, and
        // the operand ring holds up to 12 stages of two k-blocks
        const int tm_stages = (512 - a_col0) / kBK;
        ca.a_tmem = tm_stages >= 4 ? 1 : 0;
        ca.a_col0 = ca.a_tmem ? a_col0 : 0;
        if (ca.a_tmem) {
            const int n = tm_stages < 6 ? tm_stages : 6;
            const int per_raw = 2 * kQ4TileBytes + 16 + 16;
            const int per_b = 2 * ntile * kBK * 2 + 16;
            int sb = (kFullSmem - fixed0 - n * per_raw) / per_b;
            if (sb > 12) sb = 12;
            ca.tmem_cols = pow2ceil(a_col0 + n * kBK);
            ca.raw_stages = ca.stages = n;
            ca.b_stages = sb;
            ca.smem = static_cast<size_t>(fixed0) + static_cast<size_t>(n) * per_raw + static_cast<size_t>(sb) * per_b;
            return sb >= 2 && ca.smem <= static_cast<size_t>(kFullSmem);
        }
        for (int i = 0; i < 3; ++i) {
            const int fixed = fixed0 + kRaw[i] * (kQ4TileBytes + 16) + kA[i] * (static_cast<int>(kABytes) + 16);
            const int sb = (kFullSmem - fixed) / b_stage;
            if (sb >= 2 || i == 2) {
                ca.raw_stages = kRaw[i];
                ca.stages = kA[i];
                ca.b_stages = sb > 24 ? 24 : sb;
                ca.smem = static_cast<size_t>(fixed) + static_cast<size_t>(ca.b_stages) * b_stage;
                break;
            }
        }
        return ca.b_stages >= 2 && ca.smem <= static_cast<size_t>(kFullSmem);
    }
    ca.raw_stages = 0;
    ca.b_stages = 0;
    ca.a_tmem = 0;
    ca.a_col0 = 0;
    // wide residual tiles read the old residual from global memory (a warp's 32 rows of a token
    // are one 128-byte line), not from a staged copy: the ring keeps the room
    const int fixed = fixed0;
    int st = (smem_budget - fixed) / (stage_bytes + 16);
    if (st > 32) st = 32;
    if (st < 2) return false;
    ca.stages = st;
    ca.smem = static_cast<size_t>(fixed) + static_cast<size_t>(st) * (stage_bytes + 16);
    return ca.smem <= static_cast<size_t>(kFullSmem);
}

cudaError_t chain_init_attrs() {
    cudaError_t e = cudaFuncSetAttribute(reinterpret_cast<const void*>(k_chain<false>),
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, kFullSmem);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(reinterpret_cast<const void*>(k_chain<true>),
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, kFullSmem);
    return e;
}

cudaError_t chain_launch(const ChainMaps& maps, const ChainArgs& ca, cudaStream_t st, bool pdl) {
    for (int i = 0; i < ca.n_phases; ++i) {
        const GemmPlan& p = ca.ph[i].p;
        const int dr = ca.ph[i].dep_rows;
        if (p.grid > ca.grid || !ca.ph[i].partials || !ca.ph[i].tickets || (i > 0 && (dr < 0 || (dr & (dr - 1)) != 0)))
            return cudaErrorInvalidValue;
    }
    // a device-resolved row count changes a phase's tiling: no later phase may wait on its flags
    if (ca.dyn_rows && ca.n_phases != 1) return cudaErrorInvalidValue;
    if (ca.q4) {  // every phase's weights in the 4-bit tile format
        for (int i = 0; i < ca.n_phases; ++i)
            if (!ca.ph[i].w_tiles) return cudaErrorInvalidValue;
        if (ca.raw_stages < 2 || ca.raw_stages > 32 || ca.b_stages < 2 || ca.b_stages > 32) return cudaErrorInvalidValue;
        return launch_k(k_chain<true>, dim3(ca.grid), dim3(kChainThreadsQ4), ca.smem, st, pdl, maps, ca);
    }
    return launch_k(k_chain<false>, dim3(ca.grid), dim3(kChainThreads), ca.smem, st, pdl, maps, ca);
}

}  // namespace dllm
